"""Forecast parity on the values cached features can hold beyond smooth trajectories.

Eq. 13 (Sec. 3.3) is a plain weighted sum of whatever the DiT stored, so it has to carry a NaN
or an infinity in a cached feature through to the forecast, stay finite on values near the
largest bf16 / fp32 number whenever the exact combination is representable, and stay
accurate on subnormals and exact zeros.  Every case here plants such values in the history
(at tile boundaries, inside tiles and in the ragged tail of each layer), runs the CUDA path
with each kernel pinned, and checks every element against the fp64 oracle on the same stored
inputs: NaN where the oracle gives NaN, the infinity of the oracle's sign where the oracle
gives an infinity or a finite value beyond the output type's range, and otherwise the
tolerance 1e-5 (fp32 out) / 2^-8 (bf16 out) times sum_j |W_j||F_j|, plus, below the smallest
normal number, the absolute spacing of fp32 arithmetic (gpu_helpers.subnormal_floor).  The same
values go through the fused sampler update (Euler and a x + b v_hat + c z).
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2608_28670_gb300 import barycache as bc
from paper_2608_28670_gb300 import synth
from tests.gpu_helpers import (assert_close_special, empty_out, oracle_weights, stream,
                               subnormal_floor, to_device, to_host)

pytestmark = pytest.mark.gpu

KERNELS = [bc.KERNEL_REGISTER, bc.KERNEL_PIPELINE]
KNAME = {bc.KERNEL_REGISTER: "register", bc.KERNEL_PIPELINE: "pipeline"}
DT_NAME = {bc.DTYPE_F32: "f32", bc.DTYPE_BF16: "bf16"}
MODES = {bc.MODE_EXACT: "exact", bc.MODE_PAPER: "paper"}
FAMILIES = ["nonfinite", "near_max", "subnormal", "zeros"]
IO = [(bc.DTYPE_BF16, bc.DTYPE_BF16), (bc.DTYPE_F32, bc.DTYPE_F32),
      (bc.DTYPE_BF16, bc.DTYPE_F32), (bc.DTYPE_F32, bc.DTYPE_BF16)]

# Equispaced flow times, one step past the newest node: exact weights are binomial,
# (1), (2, -1), (3, -3, 1), (4, -6, 4, -1), so sum_j |W_j| = 2^K - 1.
TIMES = [0.9, 0.85, 0.8, 0.75]
T_NEW = 0.7


@pytest.fixture(scope="module", autouse=True)
def built():
    import __graft_entry__
    __graft_entry__.build_libraries()
    torch.cuda.set_device(0)


def tile_elems(dt):
    return 8192 if dt == bc.DTYPE_BF16 else 4096      # one 16 KiB tile of one slot


def layer_sizes(dt):
    T = tile_elems(dt)
    ev = 16 if dt == bc.DTYPE_BF16 else 8              # elements per 32-byte vector
    return [3 * T + 5, 2 * T + 3 * ev + 1]             # ragged ends of 5 and 1 elements


def positions(n, dt):
    """Element indices worth planting at: both sides of each 16 and 32 KiB tile boundary,
    the first element, and the ragged tail."""
    T = tile_elems(dt)
    cand = [0, 1, T - 1, T, T + 1, 2 * T - 1, 2 * T, 2 * T + 1, 3 * T - 1, n - 1, n - 2, n - 3]
    return sorted({p for p in cand if 0 <= p < n})


def to_stored(v32: np.ndarray, dt) -> np.ndarray:
    v32 = np.asarray(v32, dtype=np.float32)
    return synth.f32_to_bf16_bits(v32) if dt == bc.DTYPE_BF16 else v32


def family_values(family, n, K, dt, seed):
    """History of one layer, oldest first: K float32 arrays (stored rounding applied later)."""
    rng = np.random.default_rng(seed)
    taus = TIMES[:K]
    smooth = synth.host_trajectories([(n,)], taus, dtype="f32", degree=2, noise_std=1e-2,
                                     seed=seed)
    F = [smooth[i][0].copy() for i in range(K)]        # F[i]: oldest i = 0 ... newest K - 1
    pos = positions(n, dt)
    new, old = K - 1, 0
    if family == "nonfinite":
        inf, nan = np.float32(np.inf), np.float32(np.nan)
        for q, p in enumerate(pos):
            kind = q % 6
            if kind == 0:
                F[new][p] = nan
            elif kind == 1:
                F[old][p] = inf
            elif kind == 2:
                F[new][p] = -inf
            elif kind == 3:                             # +inf in the two newest nodes
                F[new][p] = inf
                F[max(new - 1, 0)][p] = inf
            elif kind == 4:
                F[new][p] = nan
                F[old][p] = inf
            else:
                for i in range(K):
                    F[i][p] = -inf
    elif family == "near_max":
        M = np.float32(3.0e38)
        for q, p in enumerate(pos):
            lo, hi = max(p - 20, 0), min(p + 20, n)
            sgn = 1.0 if q % 2 == 0 else -1.0
            if q % 3 == 2 and K >= 2:
                # a combination beyond the range: +3.3e38 at the newest node, -3.3e38 at
                # the others (the oracle's value decides: an infinity of its sign)
                F[new][lo:hi] = np.float32(3.3e38)
                for i in range(K - 1):
                    F[i][lo:hi] = np.float32(-3.3e38)
            else:
                # a slow trend near the maximum: the exact forecast is still representable,
                # but the plain fp32 partial sums (3 x 3e38, 4 x 3e38, ...) are not
                for i in range(K):
                    F[i][lo:hi] = np.float32(sgn * M * (1.0 + 0.01 * taus[i]))
    elif family == "subnormal":
        if dt == bc.DTYPE_BF16:
            bits = rng.integers(1, 0x80, (K, n), dtype=np.uint32) << 16
        else:
            bits = rng.integers(1, 0x800000, (K, n), dtype=np.uint32)
        bits |= (rng.integers(0, 2, (K, n), dtype=np.uint32) << 31)
        F = [bits[i].view(np.float32).copy() for i in range(K)]
    elif family == "zeros":
        sign = rng.integers(0, 2, (K, n), dtype=np.uint32) << 31
        F = [sign[i].view(np.float32).copy() for i in range(K)]
    else:
        raise ValueError(family)
    return [to_stored(f, dt) for f in F]


def make_cache(numels, K, in_dt, mode, kernel, history):
    """Cache of len(numels) layers with history[i][l] pushed oldest first at TIMES."""
    h = bc.bc_cache_create(numels, K, in_dt, bc.make_params(mode=mode))
    bc.bc_cache_set_kernel(h, kernel)
    for i in range(K):
        dev = [to_device(history[i][l]) for l in range(len(numels))]
        bc.bc_cache_push(h, [d.data_ptr() for d in dev], TIMES[i], stream())
        torch.cuda.synchronize()
    return h


@pytest.mark.parametrize("mode", list(MODES), ids=MODES.get)
@pytest.mark.parametrize("family", FAMILIES)
@pytest.mark.parametrize("io", IO, ids=lambda io: f"{DT_NAME[io[0]]}-{DT_NAME[io[1]]}")
@pytest.mark.parametrize("K", [1, 2, 3, 4])
@pytest.mark.parametrize("kernel", KERNELS, ids=KNAME.get)
def test_forecast_edge_values(kernel, K, io, family, mode):
    in_dt, out_dt = io
    numels = layer_sizes(in_dt)
    per_layer = [family_values(family, n, K, in_dt, seed=101 * l + 7 * K + in_dt)
                 for l, n in enumerate(numels)]
    history = [[per_layer[l][i] for l in range(len(numels))] for i in range(K)]
    h = make_cache(numels, K, in_dt, mode, kernel, history)
    try:
        outs = [empty_out(n, out_dt) for n in numels]
        bc.bc_forecast(h, T_NEW, [o.data_ptr() for o in outs], out_dt, stream())
        torch.cuda.synchronize()
        bc.bc_cache_check(h)
        nodes = TIMES[:K][::-1]
        W = oracle_weights(nodes, T_NEW, mode)
        floor = subnormal_floor(K, float(np.abs(W).sum()), out_dt)
        for l, n in enumerate(numels):
            F = [history[i][l] for i in range(K - 1, -1, -1)]          # newest first
            ref, bound = oracle.combine(F, W)
            assert_close_special(to_host(outs[l], out_dt), ref, bound, out_dt, floor,
                                 f"{family} layer {l}")
    finally:
        bc.bc_cache_destroy(h)


@pytest.mark.parametrize("family", FAMILIES)
@pytest.mark.parametrize("x_dt", [bc.DTYPE_F32, bc.DTYPE_BF16])
@pytest.mark.parametrize("K", [1, 2, 3, 4])
@pytest.mark.parametrize("kernel", KERNELS, ids=KNAME.get)
def test_update_branch_edge_values(kernel, K, x_dt, family):
    # Layer 0 is a block output, layer 1 the cached model output whose forecast drives the
    # sampler update; its history holds the planted values.  Both the Euler step
    # (bc_forecast_step) and the general a x + b v_hat + c z update (bc_forecast_update) run.
    in_dt = bc.DTYPE_BF16
    numels = layer_sizes(in_dt)
    v_hist = family_values(family, numels[1], K, in_dt, seed=55 + K)
    blk = synth.host_trajectories([(numels[0],)], TIMES[:K], dtype="bf16", seed=3)
    history = [[blk[i][0], v_hist[i]] for i in range(K)]
    x0 = to_stored(np.linspace(-2.0, 2.0, numels[1], dtype=np.float32), x_dt)
    z = to_stored(np.cos(np.arange(numels[1], dtype=np.float32)), x_dt)
    h = make_cache(numels, K, in_dt, bc.MODE_PAPER, kernel, history)
    try:
        W = oracle_weights(TIMES[:K][::-1], T_NEW, bc.MODE_PAPER)
        V = [history[i][1] for i in range(K - 1, -1, -1)]
        wsum = float(np.abs(W).sum())
        for kind, (a, b, c) in (("euler", (1.0, -0.05, 0.0)), ("update", (0.99, -0.05, 0.01))):
            out0 = empty_out(numels[0], bc.DTYPE_BF16)
            x = to_device(x0)
            zd = to_device(z)
            if kind == "euler":
                bc.bc_forecast_step(h, T_NEW, b, [out0.data_ptr(), None], bc.DTYPE_BF16, 1,
                                    x.data_ptr(), x_dt, stream())
                ref, _, bound = oracle.euler(V, W, x0, b)
            else:
                bc.bc_forecast_update(h, T_NEW, a, b, c, [out0.data_ptr(), None],
                                      bc.DTYPE_BF16, 1, x.data_ptr(), x_dt, zd.data_ptr(),
                                      stream())
                ref, bound = oracle.update(V, W, x0, a, b, c, z)
            torch.cuda.synchronize()
            bc.bc_cache_check(h)
            # the update adds up to three more fp32 roundings of terms of x's magnitude
            floor = abs(b) * subnormal_floor(K, wsum, bc.DTYPE_F32) + 3 * 2.0 ** -150 + (
                2.0 ** -134 if x_dt == bc.DTYPE_BF16 else 0.0)
            assert_close_special(to_host(x, x_dt), ref, bound, x_dt, floor,
                                 f"{kind} x ({family})")
            rb, bb = oracle.combine([history[i][0] for i in range(K - 1, -1, -1)], W)
            assert_close_special(to_host(out0, bc.DTYPE_BF16), rb, bb, bc.DTYPE_BF16,
                                 what=f"{kind} block output")
    finally:
        bc.bc_cache_destroy(h)


@pytest.mark.parametrize("kernel", KERNELS, ids=KNAME.get)
@pytest.mark.parametrize("dt", [bc.DTYPE_BF16, bc.DTYPE_F32])
def test_trend_near_the_maximum_stays_finite(kernel, dt):
    # Every element of a cubic-exact K = 4 window sits near the maximum: the exact weights
    # (4, -6, 4, -1) make the plain fp32 partial sums overflow (4 x 3e38), while the forecast
    # itself (the next value of a slow linear trend) is representable.  All of it must come
    # out finite and match the oracle.
    n = 4 * tile_elems(dt) + 9
    K = 4
    rng = np.random.default_rng(9)
    base = (3.0e38 * (0.97 + 0.01 * rng.random(n))).astype(np.float32)
    sign = np.where(rng.random(n) < 0.5, -1.0, 1.0).astype(np.float32)
    hist = [[to_stored(sign * base * np.float32(1.0 + 0.005 * i), dt)] for i in range(K)]
    h = make_cache([n], K, dt, bc.MODE_EXACT, kernel, hist)
    try:
        out = empty_out(n, dt)
        bc.bc_forecast(h, T_NEW, [out.data_ptr()], dt, stream())
        torch.cuda.synchronize()
        W = oracle_weights(TIMES[::-1], T_NEW, bc.MODE_EXACT)
        ref, bound = oracle.combine([hist[i][0] for i in range(K - 1, -1, -1)], W)
        assert np.all(np.isfinite(ref))
        got = to_host(out, dt)
        assert_close_special(got, ref, bound, dt, what="near-maximum trend")
        g = got if dt == bc.DTYPE_F32 else synth.bf16_bits_to_f32(got)
        assert np.all(np.isfinite(g))
    finally:
        bc.bc_cache_destroy(h)
