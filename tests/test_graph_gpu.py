"""A whole sampling loop captured into one CUDA graph and replayed.

Pushes (zero-copy slots and commits), forecasts and the fused DDIM update enqueue only
kernels on the caller's stream (no allocation, copy or synchronisation), so a loop of them
can be captured.  The graph holds the slot addresses and weights that the calls chose while
it was captured; replaying it repeats that device work (the handle's host state does not
move).  The replay must reproduce the eager loop bit for bit, every time, and the eager
loop must match the fp64 oracle replayed step by step.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2608_28670_gb300 import barycache as bc
from paper_2608_28670_gb300 import synth
from tests.gpu_helpers import device_view

pytestmark = pytest.mark.gpu

STEPS, INTERVAL, K = 20, 3, 3
NUMELS = [2 * 256 * 1152, 2 * 4 * 32 * 32]      # a block output + the eps prediction


@pytest.fixture(scope="module", autouse=True)
def built():
    import __graft_entry__
    __graft_entry__.build_libraries()
    torch.cuda.set_device(0)


def schedule():
    ts = [980.0 - 20.0 * i for i in range(STEPS)]
    betas = np.linspace(1e-4, 0.02, 1000)
    ab = np.cumprod(1.0 - betas)
    coef = []
    for i in range(STEPS):
        t, t_prev = int(ts[i]), int(ts[i]) - 20
        coef.append(bc.bc_ddim_coefficients(ab[t], ab[t_prev] if t_prev >= 0 else 1.0, 0.0))
    return ts, coef


def run_loop(h, x, out, sched, ts, coef, s):
    """One DDIM sampling run: full steps have the stand-in write both layers into the next
    slot and take the DDIM step from the written eps; skipped steps forecast both layers and
    take the fused DDIM step."""
    for i in range(STEPS):
        a, b, _ = coef[i]
        if sched[i]:
            slots = bc.bc_cache_next_slot_ptrs(h, 2)
            for l, n in enumerate(NUMELS):
                synth.fill_device(slots[l], bc.DTYPE_F32, n, seed=5, tensor_id=l, step_id=i,
                                  tau=ts[i] / 1000.0, degree=2, noise_std=1e-3, stream=s)
            bc.bc_cache_commit(h, ts[i])
            x.mul_(a).add_(device_view(slots[1], NUMELS[1], bc.DTYPE_F32), alpha=b)
        else:
            bc.bc_forecast_update(h, ts[i], a, b, 0.0, [out.data_ptr(), None], bc.DTYPE_F32, 1,
                                  x.data_ptr(), bc.DTYPE_F32, None, s)


def test_graph_replay_equals_eager_loop_and_oracle():
    ts, coef = schedule()
    sched = bc.bc_schedule_equal(STEPS, INTERVAL, K)
    x0 = torch.linspace(-1.0, 1.0, NUMELS[1], device="cuda")
    h = bc.bc_cache_create(NUMELS, K, bc.DTYPE_F32)
    try:
        out = torch.empty(NUMELS[0], device="cuda")
        x = x0.clone()
        s = torch.cuda.current_stream().cuda_stream
        run_loop(h, x, out, sched, ts, coef, s)                # eager (also warms up)
        torch.cuda.synchronize()
        x_eager, out_eager = x.clone(), out.clone()

        # fp64 oracle replay of the same loop from the generator's stored values
        slot_hist, x_ref = [], x0.double().cpu().numpy()
        for i in range(STEPS):
            a, b, _ = coef[i]
            if sched[i]:
                v = torch.empty(NUMELS[1], device="cuda")
                synth.fill_device(v.data_ptr(), bc.DTYPE_F32, NUMELS[1], seed=5, tensor_id=1,
                                  step_id=i, tau=ts[i] / 1000.0, degree=2, noise_std=1e-3,
                                  stream=s)
                torch.cuda.synchronize()
                slot_hist.append((ts[i], v.cpu().numpy()))
                x_ref = a * x_ref + b * slot_hist[-1][1].astype(np.float64)
            else:
                win = slot_hist[-K:][::-1]
                W = oracle.paper_weights([w[0] for w in win], ts[i])
                v_hat, _ = oracle.combine([w[1] for w in win], W)
                x_ref = a * x_ref + b * v_hat
        np.testing.assert_allclose(x_eager.cpu().numpy(), x_ref, rtol=1e-4, atol=1e-4)

        bc.bc_cache_reset(h)
        g = torch.cuda.CUDAGraph()
        x.copy_(x0)
        torch.cuda.synchronize()
        with torch.cuda.graph(g, capture_error_mode="thread_local"):
            run_loop(h, x, out, sched, ts, coef, torch.cuda.current_stream().cuda_stream)
        for _ in range(2):
            x.copy_(x0)
            out.zero_()
            g.replay()
            torch.cuda.synchronize()
            assert torch.equal(x, x_eager)
            assert torch.equal(out, out_eager)
        bc.bc_cache_check(h)
    finally:
        bc.bc_cache_destroy(h)


@pytest.mark.parametrize("kernel", [bc.KERNEL_REGISTER, bc.KERNEL_PIPELINE])
def test_probe_drift_replays_from_a_graph(kernel):
    # The adaptive schedule's probe drift (handle and no-allocation forms) enqueues kernels
    # only, so it can be captured: a replay computes from the probe tensors' current contents,
    # bit for bit the eager call on the same contents, and both match the fp64 oracle.
    n = 600_001                                    # ragged: a tail shorter than one group
    rng = np.random.default_rng(7)
    prev_h = rng.standard_normal(n).astype(np.float32)
    cur_h = prev_h + 0.05 * rng.standard_normal(n).astype(np.float32)
    cur, prev = torch.from_numpy(cur_h).cuda(), torch.from_numpy(prev_h).cuda()
    f64 = dict(dtype=torch.float64, device="cuda")
    h = bc.bc_cache_create([16], 2, bc.DTYPE_F32)
    bc.bc_cache_set_kernel(h, kernel)
    s = torch.cuda.current_stream().cuda_stream

    def eager():
        o, o_na = torch.zeros(3, **f64), torch.zeros(3, **f64)
        bc.bc_probe_drift(h, cur.data_ptr(), prev.data_ptr(), n, bc.DTYPE_F32, o.data_ptr(), s)
        bc.bc_probe_drift_noalloc(cur.data_ptr(), prev.data_ptr(), n, bc.DTYPE_F32,
                                  o_na.data_ptr(), s)
        torch.cuda.synchronize()
        return o, o_na

    try:
        e, e_na = eager()                          # also the first, uncaptured calls
        out, out_na = torch.full((3,), -1.0, **f64), torch.full((3,), -1.0, **f64)
        g = torch.cuda.CUDAGraph()
        side = torch.cuda.Stream()
        with torch.cuda.stream(side):
            l0 = bc.bc_cache_stats(h)["kernel_launches"]
            with torch.cuda.graph(g, stream=side, capture_error_mode="thread_local"):
                bc.bc_probe_drift(h, cur.data_ptr(), prev.data_ptr(), n, bc.DTYPE_F32,
                                  out.data_ptr(), side.cuda_stream)
                bc.bc_probe_drift_noalloc(cur.data_ptr(), prev.data_ptr(), n, bc.DTYPE_F32,
                                          out_na.data_ptr(), side.cuda_stream)
            assert bc.bc_cache_stats(h)["kernel_launches"] - l0 == 2
        g.replay()
        torch.cuda.synchronize()
        assert torch.equal(out, e) and torch.equal(out_na, e_na)
        np.testing.assert_allclose(out.cpu().numpy(), oracle.drift(cur_h, prev_h), rtol=2e-6)
        np.testing.assert_allclose(out_na.cpu().numpy(), oracle.drift(cur_h, prev_h), rtol=2e-6)
        cur.mul_(2.0)                              # new contents: the replay must read them
        cur_h = cur_h * np.float32(2.0)
        torch.cuda.synchronize()
        g.replay()
        torch.cuda.synchronize()
        e2, e2_na = eager()
        assert torch.equal(out, e2) and torch.equal(out_na, e2_na)
        assert not torch.equal(out, e)
        np.testing.assert_allclose(out.cpu().numpy(), oracle.drift(cur_h, prev_h), rtol=2e-6)
        bc.bc_cache_check(h)
    finally:
        torch.cuda.synchronize()
        bc.bc_cache_destroy(h)


@pytest.mark.parametrize("kernel", [bc.KERNEL_REGISTER, bc.KERNEL_PIPELINE])
def test_pushes_replay_from_a_graph(kernel):
    # A push over more layers than a parameter block holds (split into parameter-block launches
    # while captured) and a flat push of a slot image, captured into one graph: each replay
    # copies the sources' current bytes into the slots chosen while capturing.
    n_l, n = 2048, 2048
    K = 3
    h = bc.bc_cache_create([n] * n_l, K, bc.DTYPE_BF16)
    bc.bc_cache_set_kernel(h, kernel)
    s = torch.cuda.current_stream().cuda_stream
    try:
        offs = bc.bc_cache_layout(h)
        src = torch.randint(-32768, 32767, (n * n_l,), dtype=torch.int16, device="cuda")
        img = torch.randint(-32768, 32767, (offs[-1] // 2,), dtype=torch.int16, device="cuda")
        ptrs = np.array([src.data_ptr() + 2 * n * l for l in range(n_l)], dtype=np.uint64)
        bc.bc_cache_push(h, ptrs, 0.9, s)          # first uses outside the capture
        bc.bc_cache_push_flat(h, img.data_ptr(), 0.8, s)
        torch.cuda.synchronize()
        g = torch.cuda.CUDAGraph()
        side = torch.cuda.Stream()
        with torch.cuda.stream(side):
            l0 = bc.bc_cache_stats(h)["kernel_launches"]
            with torch.cuda.graph(g, stream=side, capture_error_mode="thread_local"):
                bc.bc_cache_push(h, ptrs, 0.7, side.cuda_stream)
                bc.bc_cache_push_flat(h, img.data_ptr(), 0.6, side.cuda_stream)
            assert bc.bc_cache_stats(h)["kernel_launches"] - l0 == 4    # 1016 + 1016 + 16, 1
        # slots chosen while capturing: 0.7 went to node 1's slot, 0.6 to node 0's
        per_layer_slot = bc.bc_cache_slot_ptrs(h, 1)[0]
        flat_slot = bc.bc_cache_slot_ptrs(h, 0)[0]
        for _ in range(2):
            src.add_(1)
            img.sub_(3)
            torch.cuda.synchronize()
            g.replay()
            torch.cuda.synchronize()
            got = device_view(per_layer_slot, n * n_l, bc.DTYPE_BF16)
            assert torch.equal(got, src)
            got = device_view(flat_slot, offs[-1] // 2, bc.DTYPE_BF16)
            assert torch.equal(got, img)
        bc.bc_cache_check(h)
    finally:
        torch.cuda.synchronize()
        bc.bc_cache_destroy(h)
