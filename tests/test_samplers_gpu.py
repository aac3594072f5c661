"""GPU parity of the sampler update (DDPM / DDIM / Euler), the flat many-tensor forecast, the
probe drift of the adaptive schedule, and an end-to-end sampling loop over a schedule.

Coefficients passed to the library come from the oracle (so no expected value depends on the
library); the library's own coefficient helpers are checked against the oracle on the CPU.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2608_28670_gb300 import barycache as bc
from paper_2608_28670_gb300 import synth
from tests.gpu_helpers import (assert_close, device_view, empty_out, stream, to_device,
                               to_host)

pytestmark = pytest.mark.gpu
DT = {bc.DTYPE_F32: "f32", bc.DTYPE_BF16: "bf16"}


@pytest.fixture(scope="module", autouse=True)
def built():
    import __graft_entry__
    __graft_entry__.build_libraries()
    torch.cuda.set_device(0)


def _cache_with(numels, times, in_dt, seed, K=3, kernel=bc.KERNEL_AUTO):
    feats = synth.host_trajectories([(n,) for n in numels], times, dtype=DT[in_dt], seed=seed)
    h = bc.bc_cache_create(numels, K, in_dt)
    bc.bc_cache_set_kernel(h, kernel)
    for t, per in zip(times, feats):
        dev = [to_device(f) for f in per]
        bc.bc_cache_push(h, [d.data_ptr() for d in dev], t, stream())
        torch.cuda.synchronize()
    return h, feats


@pytest.mark.parametrize("kernel", [bc.KERNEL_REGISTER, bc.KERNEL_PIPELINE])
@pytest.mark.parametrize("kind", ["ddpm", "ddim0", "ddim1"])
@pytest.mark.parametrize("x_dt", [bc.DTYPE_F32, bc.DTYPE_BF16])
@pytest.mark.parametrize("with_z", [False, True])
def test_update_matches_oracle(kind, x_dt, with_z, kernel):
    # DDIM-style integer timesteps; eps is the cached model output (layer 1).
    numels = [3 * 8192 + 11, 65_536 + 3]
    times = [980.0, 960.0, 940.0]
    t_new = 920.0
    h, feats = _cache_with(numels, times, bc.DTYPE_BF16, seed=31, kernel=kernel)
    try:
        betas = np.linspace(1e-4, 0.02, 1000)
        ab = np.cumprod(1 - betas)
        if kind == "ddpm":
            a, b, c = oracle.ddpm_coefficients(1 - betas[920], ab[920])
        else:
            a, b, c = oracle.ddim_coefficients(ab[920], ab[900], 0.0 if kind == "ddim0" else 1.0)
        x0 = synth.host_trajectories([(numels[1],)], [0.0], dtype=DT[x_dt], degree=0,
                                     noise_std=0.0, seed=32)[0][0]
        z0 = synth.host_trajectories([(numels[1],)], [0.0], dtype=DT[x_dt], degree=0,
                                     noise_std=0.0, seed=33)[0][0]
        x = to_device(x0)
        z = to_device(z0) if with_z else None
        out0 = empty_out(numels[0], bc.DTYPE_BF16)
        bc.bc_forecast_update(h, t_new, a, b, c, [out0.data_ptr(), None], bc.DTYPE_BF16, 1,
                              x.data_ptr(), x_dt, z.data_ptr() if with_z else None, stream())
        torch.cuda.synchronize()
        W = oracle.paper_weights([940.0, 960.0, 980.0], t_new)
        nf = feats[::-1]
        ref, bound = oracle.combine([f[0] for f in nf], W)
        assert_close(to_host(out0, bc.DTYPE_BF16), ref, bound, bc.DTYPE_BF16, "block")
        x_ref, xb = oracle.update([f[1] for f in nf], W, x0, a, b, c if with_z else 0.0,
                                  z0 if with_z else None)
        assert_close(to_host(x, x_dt), x_ref, xb, x_dt, f"{kind} x")
    finally:
        bc.bc_cache_destroy(h)


def test_update_rejects_aliasing_and_bad_coefficients():
    h, _ = _cache_with([4096], [0.9, 0.8, 0.7], bc.DTYPE_F32, seed=1)
    try:
        x = torch.zeros(4096, device="cuda")
        with pytest.raises(bc.BaryCacheError) as ei:
            bc.bc_forecast_update(h, 0.6, 1.0, 0.1, 0.2, [None], bc.DTYPE_F32, 0, x.data_ptr(),
                                  bc.DTYPE_F32, x.data_ptr(), stream())
        assert ei.value.status == bc.ERR_INVALID_ARG          # z aliases x
        with pytest.raises(bc.BaryCacheError) as ei:
            bc.bc_forecast_update(h, 0.6, float("inf"), 0.1, 0.0, [None], bc.DTYPE_F32, 0,
                                  x.data_ptr(), bc.DTYPE_F32, None, stream())
        assert ei.value.status == bc.ERR_INVALID_ARG
        with pytest.raises(bc.BaryCacheError) as ei:
            bc.bc_forecast_update(h, 0.6, 1.0, 0.1, 0.2, [None], bc.DTYPE_F32, 0, x.data_ptr(),
                                  bc.DTYPE_F32, x.data_ptr() + 4, stream())
        assert ei.value.status == bc.ERR_ALIGNMENT
    finally:
        bc.bc_cache_destroy(h)


@pytest.mark.parametrize("kernel", [bc.KERNEL_REGISTER, bc.KERNEL_PIPELINE])
@pytest.mark.parametrize("in_dt", [bc.DTYPE_BF16, bc.DTYPE_F32])
def test_flat_forecast_many_small_tensors(in_dt, kernel):
    rng = np.random.default_rng(5)
    numels = [int(v) for v in rng.integers(1, 3000, 500)] + [0, 40_000]
    times = [0.9, 0.85, 0.8]
    h, feats = _cache_with(numels, times, in_dt, seed=6, kernel=kernel)
    try:
        offs = bc.bc_cache_layout(h, len(numels))
        assert offs[-1] * 3 == bc.bc_cache_bytes(h)
        eb = 2 if in_dt == bc.DTYPE_BF16 else 4
        flat = torch.empty(offs[-1] // eb, dtype=torch.int16 if eb == 2 else torch.float32,
                           device="cuda")
        s0 = bc.bc_cache_stats(h)["kernel_launches"]
        bc.bc_forecast_flat(h, 0.75, flat.data_ptr(), stream())
        torch.cuda.synchronize()
        assert bc.bc_cache_stats(h)["kernel_launches"] - s0 == 1
        # the per-layer path (one launch with a 502-entry layer table) gives the same bits
        outs = [empty_out(n, in_dt) for n in numels]
        bc.bc_forecast(h, 0.75, [o.data_ptr() if n else None for o, n in zip(outs, numels)],
                       in_dt, stream())
        torch.cuda.synchronize()
        host = to_host(flat, in_dt)
        W = oracle.paper_weights([0.8, 0.85, 0.9], 0.75)
        nf = feats[::-1]
        for l, n in enumerate(numels):
            if n == 0:
                continue
            got = host[offs[l] // eb: offs[l] // eb + n]
            np.testing.assert_array_equal(got, to_host(outs[l], in_dt))
            if l % 25 == 0 or l >= len(numels) - 2:
                ref, bound = oracle.combine([f[l] for f in nf], W)
                assert_close(got, ref, bound, in_dt, f"flat layer {l}")
    finally:
        bc.bc_cache_destroy(h)


def test_flat_forecast_rejects_bad_output():
    h, _ = _cache_with([100, 200], [0.9, 0.8], bc.DTYPE_F32, seed=2)
    try:
        slot = bc.bc_cache_slot_ptrs(h, 0, 2)[0]
        with pytest.raises(bc.BaryCacheError) as ei:
            bc.bc_forecast_flat(h, 0.7, slot, stream())
        assert ei.value.status == bc.ERR_INVALID_ARG
        buf = torch.empty(1024, device="cuda")
        with pytest.raises(bc.BaryCacheError) as ei:
            bc.bc_forecast_flat(h, 0.7, buf.data_ptr() + 8, stream())
        assert ei.value.status == bc.ERR_ALIGNMENT
    finally:
        bc.bc_cache_destroy(h)


@pytest.mark.parametrize("kernel", [bc.KERNEL_REGISTER, bc.KERNEL_PIPELINE],
                         ids=["register", "pipeline"])
@pytest.mark.parametrize("dt", [bc.DTYPE_BF16, bc.DTYPE_F32])
@pytest.mark.parametrize("n", [0, 1, 7, 8, 9, 1000, 123_457, 8192 * 37 + 11,
                               4 * 1024 * 1024 + 3])
def test_probe_drift_matches_oracle_and_is_deterministic(dt, n, kernel):
    # The pipeline form stages 16 KiB tiles of both tensors (8192 bf16 / 4096 fp32
    # elements); these sizes give one partial tile, many tiles with a ragged last one, and
    # an element tail shorter than one 16-byte group.
    rng = np.random.default_rng(n + dt)
    prev = rng.standard_normal(n).astype(np.float32)
    cur = prev + 0.05 * rng.standard_normal(n).astype(np.float32)
    if dt == bc.DTYPE_BF16:
        prev, cur = synth.f32_to_bf16_bits(prev), synth.f32_to_bf16_bits(cur)
    h = bc.bc_cache_create([16], 2, bc.DTYPE_BF16)
    bc.bc_cache_set_kernel(h, kernel)
    try:
        c, p = to_device(cur), to_device(prev)
        out = torch.full((2, 3), -1.0, dtype=torch.float64, device="cuda")
        for k in range(2):
            bc.bc_probe_drift(h, c.data_ptr(), p.data_ptr(), n, dt, out[k].data_ptr(), stream())
        torch.cuda.synchronize()
        got = out.cpu().numpy()
        assert np.array_equal(got[0], got[1], equal_nan=True)       # reproducible
        ref = oracle.drift(cur, prev)
        if n == 0:
            assert list(got[0]) == [0.0, 0.0, 0.0]
        else:
            np.testing.assert_allclose(got[0], ref, rtol=2e-6)
        bc.bc_cache_check(h)
    finally:
        bc.bc_cache_destroy(h)


@pytest.mark.parametrize("kernel", [bc.KERNEL_REGISTER, bc.KERNEL_PIPELINE],
                         ids=["register", "pipeline"])
def test_probe_drift_special_values(kernel):
    h = bc.bc_cache_create([16], 2, bc.DTYPE_BF16)
    bc.bc_cache_set_kernel(h, kernel)
    try:
        z = torch.zeros(1000, device="cuda")
        o = torch.ones(1000, device="cuda")
        out = torch.empty(3, dtype=torch.float64, device="cuda")
        bc.bc_probe_drift(h, o.data_ptr(), z.data_ptr(), 1000, bc.DTYPE_F32, out.data_ptr(),
                          stream())
        torch.cuda.synchronize()
        assert out.cpu().tolist() == [1000.0, 0.0, float("inf")]
        bc.bc_probe_drift(h, o.data_ptr(), o.data_ptr(), 1000, bc.DTYPE_F32, out.data_ptr(),
                          stream())
        torch.cuda.synchronize()
        assert out.cpu().tolist() == [0.0, 1000.0, 0.0]
        zn = z.clone()
        zn[500] = float("nan")
        bc.bc_probe_drift(h, z.data_ptr(), zn.data_ptr(), 1000, bc.DTYPE_F32, out.data_ptr(),
                          stream())
        torch.cuda.synchronize()
        assert np.isnan(out.cpu().numpy()).all()        # NaN, never "no change"
        with pytest.raises(bc.BaryCacheError) as ei:
            bc.bc_probe_drift(h, o.data_ptr() + 4, z.data_ptr(), 10, bc.DTYPE_F32,
                              out.data_ptr(), stream())
        assert ei.value.status == bc.ERR_ALIGNMENT
    finally:
        bc.bc_cache_destroy(h)


@pytest.mark.parametrize("adaptive", [False, True])
def test_sampling_loop_over_a_schedule(adaptive):
    """A 28-step flow sampler: full steps write the stand-in model's features into the next
    slot (zero-copy) and take the Euler step themselves; skipped steps forecast every cached
    tensor and take the fused Euler step.  Every forecast is checked against the oracle, and
    the final latent against an fp64 replay of the same loop."""
    steps, K = 28, 3
    ts = [1.0 - i / steps for i in range(steps)] + [0.0]
    numels = [20_000, 4096]                       # one block output + the velocity
    h = bc.bc_cache_create(numels, K, bc.DTYPE_BF16)
    try:
        x = torch.zeros(numels[1], dtype=torch.float32, device="cuda")
        x_ref = np.zeros(numels[1])
        out0 = empty_out(numels[0], bc.DTYPE_BF16)
        st = bc.bc_adaptive_init(0.06, K) if adaptive else None
        sched = bc.bc_schedule_equal(steps, 3, K)
        stored = []                               # host copies of pushed features, oldest first
        probe_prev = None
        n_full = 0
        for i in range(steps):
            t, dt = ts[i], ts[i + 1] - ts[i]
            # one fixed seed: the same per-element trajectories, evaluated at this step's t
            feats = synth.host_trajectories([(n,) for n in numels], [t], dtype="bf16",
                                            noise_std=1e-3, seed=100)[0]
            if adaptive:
                probe = synth.bf16_bits_to_f32(feats[1]).astype(np.float64)
                drift = 0.0 if probe_prev is None else \
                    float(np.abs(probe - probe_prev).sum() / np.abs(probe_prev).sum())
                probe_prev = probe
                full = bc.bc_adaptive_decide(st, drift)
            else:
                full = sched[i]
            if full:
                n_full += 1
                slots = bc.bc_cache_next_slot_ptrs(h, 2)
                for l, n in enumerate(numels):
                    device_view(slots[l], n, bc.DTYPE_BF16).copy_(to_device(feats[l]))
                bc.bc_cache_commit(h, t)
                stored.append((t, feats))
                v = torch.from_numpy(synth.bf16_bits_to_f32(feats[1])).cuda()
                x += dt * v
                x_ref += dt * synth.bf16_bits_to_f32(feats[1]).astype(np.float64)
            else:
                bc.bc_forecast_step(h, t, dt, [out0.data_ptr(), None], bc.DTYPE_BF16, 1,
                                    x.data_ptr(), bc.DTYPE_F32, stream())
                window = stored[-K:][::-1]
                W = oracle.paper_weights([w[0] for w in window], t)
                ref, bound = oracle.combine([w[1][0] for w in window], W)
                torch.cuda.synchronize()
                assert_close(to_host(out0, bc.DTYPE_BF16), ref, bound, bc.DTYPE_BF16,
                             f"step {i}")
                v_hat, _ = oracle.combine([w[1][1] for w in window], W)
                x_ref += dt * v_hat
        torch.cuda.synchronize()
        if not adaptive:
            assert n_full == sum(sched) == 12
        assert 0 < n_full < steps
        np.testing.assert_allclose(x.cpu().numpy(), x_ref, rtol=1e-4, atol=1e-4)
        assert bc.bc_cache_stats(h)["forecasts"] == steps - n_full
    finally:
        bc.bc_cache_destroy(h)
