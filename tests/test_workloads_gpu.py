"""Full-size parity of the five workloads, in the launch configuration the benchmark times.

The history slots are written in place by the seeded device generator (never by the
forecast path); the forecast runs through the C ABI exactly as in ``bench.py``; then every
element of the output is checked against the fp64 oracle, layer by layer, for the four
image workloads (up to 807 M elements), and for the video workload every element of three
layers per checked window plus, on every other layer, a sample of element indices (first,
last, tile boundaries and random positions).
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2608_28670_gb300 import barycache as bc
from paper_2608_28670_gb300.configs import WORKLOADS, T2V_HBM_BUDGET
from paper_2608_28670_gb300.runner import WorkloadRun
from tests.gpu_helpers import as_f64, assert_close, device_view, oracle_weights, stream

pytestmark = pytest.mark.gpu
SAMPLES = 4096


@pytest.fixture(scope="module", autouse=True)
def built():
    import __graft_entry__
    __graft_entry__.build_libraries()
    torch.cuda.set_device(0)


def sample_indices(n: int, rng) -> torch.Tensor:
    fixed = [0, 1, n // 2, n - 2, n - 1] + [min(n - 1, k * 8192 + d) for k in (1, 2, 3)
                                               for d in (-1, 0, 1)]
    idx = np.unique(np.concatenate([np.array(fixed), rng.integers(0, n, SAMPLES)]))
    return torch.from_numpy(idx[(idx >= 0) & (idx < n)]).cuda()


def gather(ptr: int, n: int, dtype: int, idx: torch.Tensor) -> np.ndarray:
    v = device_view(ptr, n, dtype)[idx]
    a = v.cpu().numpy()
    return a.view(np.uint16) if dtype == bc.DTYPE_BF16 else a


def check_run(run: WorkloadRun, rng, calls=None, full=lambda l: True, mode=bc.MODE_PAPER):
    w, h = run.w, run.h
    p = run.problem
    W = oracle_weights(list(p.nodes), p.t, mode)
    assert bc.bc_cache_nodes(h) == list(p.nodes)
    m = len(p.nodes)
    slot_ptrs = [bc.bc_cache_slot_ptrs(h, j, len(run.numels)) for j in range(m)]
    calls = range(run.calls) if calls is None else calls
    if run.euler:
        x_before = run.x.clone()
    out_dt = bc.DTYPE_BF16 if run.out_dtype == bc.DTYPE_BF16 else bc.DTYPE_F32
    for c in calls:
        run.forecast_call(c)
        torch.cuda.synchronize()
        for i in range(run.window):
            l = c * run.window + i
            if l >= run.n_feat:
                break
            n = run.numels[l]
            outv = run.outs[i].view(torch.int16) if out_dt == bc.DTYPE_BF16 else run.outs[i]
            if full(l):                  # every element of the layer
                F = [device_view(slot_ptrs[j][l], n, w.dtype).cpu().numpy() for j in range(m)]
                F = [f.view(np.uint16) if w.dtype == bc.DTYPE_BF16 else f for f in F]
                got = outv[:n].cpu().numpy()
            else:
                idx = sample_indices(n, rng)
                F = [gather(slot_ptrs[j][l], n, w.dtype, idx) for j in range(m)]
                got = outv[idx].cpu().numpy()
            ref, bound = oracle.combine(F, W)
            got = got.view(np.uint16) if out_dt == bc.DTYPE_BF16 else got
            assert_close(got, ref, bound, out_dt, f"{w.name} layer {l}")
            del F, ref, bound, got
        if run.euler and c == 0:
            nv = run.numels[-1]
            idx = torch.arange(nv, device="cuda")
            V = [gather(slot_ptrs[j][-1], nv, w.dtype, idx) for j in range(m)]
            x_ref, _, xb = oracle.euler(V, W, x_before.cpu().numpy(), p.dt)
            assert_close(run.x.cpu().numpy(), x_ref, xb, bc.DTYPE_F32, f"{w.name} Euler x")
    bc.bc_cache_check(h)            # no forecast launch gave up waiting


def test_c2i_256_every_element():
    w = WORKLOADS["c2i-256"]
    run = WorkloadRun(w, stream=stream())
    try:
        run.forecast()
        torch.cuda.synchronize()
        p = run.problem
        assert p.nodes == (940.0, 960.0, 980.0) and p.t == 920.0
        W = oracle_weights(list(p.nodes), p.t, bc.MODE_PAPER)
        n = w.layer_numel
        F = [device_view(bc.bc_cache_slot_ptrs(run.h, j, 1)[0], n, w.dtype).cpu().numpy()
             for j in range(3)]
        ref, bound = oracle.combine(F, W)
        assert_close(run.outs[0].cpu().numpy(), ref, bound, bc.DTYPE_F32, "c2i-256")
        # Exact mode recovers the quadratic trajectory: W = (3, -3, 1) exactly.
        bc.bc_cache_set_params(run.h, bc.make_params(mode=bc.MODE_EXACT))
        assert bc.bc_coefficients(run.h, 920.0) == [3.0, -3.0, 1.0]
    finally:
        run.close()


@pytest.mark.parametrize("name", ["c2i-512", "t2i-1024", "mmdit-t2i", "blockwise"])
def test_image_workloads_every_element(name):
    # (blockwise: 4096 tensors, one launch through the device layer table)
    torch.cuda.empty_cache()
    run = WorkloadRun(WORKLOADS[name], stream=stream())
    try:
        assert run.calls == 1
        check_run(run, np.random.default_rng(len(name)))
        st = run.stats()
        assert st["kernel_launches"] == 1 and st["forecasts"] == 1
        assert st["table_uploads"] == (1 if run.n_feat > 1016 else 0)
    finally:
        run.close()
        torch.cuda.empty_cache()


@pytest.mark.parametrize("name,out_dtype,mode", [
    ("mmdit-t2i", bc.DTYPE_F32, bc.MODE_PAPER),     # fp32 outputs beside the fused Euler step
    ("c2i-512", bc.DTYPE_BF16, bc.MODE_EXACT),      # exact barycentric weights, H = 4
    ("t2i-1024", bc.DTYPE_F32, bc.MODE_EXACT),
], ids=["mmdit-f32-paper", "c2i512-bf16-exact", "t2i-f32-exact"])
def test_image_workloads_other_weights_and_output_dtypes(name, out_dtype, mode):
    torch.cuda.empty_cache()
    run = WorkloadRun(WORKLOADS[name], out_dtype=out_dtype, params=bc.make_params(mode=mode),
                      stream=stream())
    try:
        check_run(run, np.random.default_rng(7), mode=mode)
    finally:
        run.close()
        torch.cuda.empty_cache()


@pytest.mark.parametrize("K", [2, 3, 4])
def test_t2v_within_budget(K):
    torch.cuda.empty_cache()
    free, _ = torch.cuda.mem_get_info()
    w = WORKLOADS["t2v"]
    if free < w.cache_bytes(K) + 8 * 10**9:
        pytest.skip(f"needs {w.cache_bytes(K) / 1e9:.0f} GB free, have {free / 1e9:.0f} GB")
    run = WorkloadRun(w, K=K, budget_bytes=T2V_HBM_BUDGET, stream=stream())
    try:
        total = bc.bc_cache_bytes(run.h) + run.window * w.layer_numel * 2
        assert total <= T2V_HBM_BUDGET
        if K <= 3:
            assert run.calls == 1
        calls = sorted({0, run.calls // 2, run.calls - 1})
        # every element of the first, a middle and the last layer of each checked window
        full = {l for c in calls for l in (c * run.window,
                                            c * run.window + (run.window - 1) // 2,
                                            min(run.n_feat, (c + 1) * run.window) - 1)}
        check_run(run, np.random.default_rng(K), calls=calls, full=lambda l: l in full)
    finally:
        run.close()
        torch.cuda.empty_cache()
