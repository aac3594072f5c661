"""Helpers shared by the GPU tests: device views of raw addresses and small parity runs."""
from __future__ import annotations

import numpy as np
import torch

import oracle
from paper_2608_28670_gb300 import barycache as bc
from paper_2608_28670_gb300 import synth
from paper_2608_28670_gb300.runner import device_view  # noqa: F401  (re-exported)

TOL = {bc.DTYPE_F32: 1e-5, bc.DTYPE_BF16: 2.0 ** -8}


def to_device(a: np.ndarray) -> torch.Tensor:
    a = np.ascontiguousarray(a).reshape(-1)
    if a.dtype == np.uint16:
        return torch.from_numpy(a.view(np.int16)).cuda()
    return torch.from_numpy(a).cuda()


def to_host(t: torch.Tensor, dtype: int) -> np.ndarray:
    a = t.detach().cpu().numpy()
    return a.view(np.uint16) if dtype == bc.DTYPE_BF16 else a


def empty_out(n: int, dtype: int, pad: int = 0) -> torch.Tensor:
    tdt = torch.float32 if dtype == bc.DTYPE_F32 else torch.int16
    return torch.empty(n + 2 * pad, dtype=tdt, device="cuda")


def as_f64(a: np.ndarray) -> np.ndarray:
    if a.dtype == np.uint16:
        return synth.bf16_bits_to_f32(a).astype(np.float64)
    return a.astype(np.float64)


def oracle_weights(nodes, t, mode, lam=0.0, delta=None, C=10.0, eta=1e-12):
    if mode == bc.MODE_EXACT:
        return oracle.lagrange(nodes, t)
    return oracle.paper_weights(nodes, t, delta=delta, lam=lam, C=C, eta=eta)


def assert_close(gpu: np.ndarray, ref: np.ndarray, bound: np.ndarray, out_dtype: int,
                 what: str = "") -> None:
    g = as_f64(gpu)
    err = np.abs(g - ref)
    tol = TOL[out_dtype] * bound
    bad = ~(err <= tol)
    if bad.any():
        i = int(np.flatnonzero(bad)[0])
        raise AssertionError(f"{what}: {bad.sum()} of {bad.size} elements off; first at {i}: "
                             f"gpu {g[i]!r} oracle {ref[i]!r} bound {bound[i]!r}")


def stream() -> int:
    return torch.cuda.current_stream().cuda_stream


# Largest finite value of each output type, and half the spacing of its subnormals.
FINITE_MAX = {bc.DTYPE_F32: float(np.finfo(np.float32).max),
              bc.DTYPE_BF16: float(synth.bf16_bits_to_f32(np.array([0x7F7F], np.uint16))[0])}
HALF_SUBNORMAL_SPACING = {bc.DTYPE_F32: 2.0 ** -150, bc.DTYPE_BF16: 2.0 ** -134}


def subnormal_floor(K: int, wsum: float, out_dtype: int) -> float:
    """Absolute error allowance below the smallest normal number.

    There fp32 has a fixed spacing of 2^-149, so each rounding of the kernel's fp32 chain can
    err by 2^-150 whatever the magnitude, and a relative bound cannot hold.  The chain has K
    roundings of terms scaled by 1/s (s < 2 sum_j |W_j|, the power of two the weights are
    divided by), undone by one multiplication by s, plus one rounding of that product; a bf16
    output then rounds once more, by at most half its own subnormal spacing (2^-134)."""
    return 2.0 ** -150 * (2 * K * wsum + 1) + (HALF_SUBNORMAL_SPACING[out_dtype]
                                               if out_dtype == bc.DTYPE_BF16 else 0.0)


def assert_close_special(gpu: np.ndarray, ref: np.ndarray, bound: np.ndarray, out_dtype: int,
                         floor: float = 0.0, what: str = "") -> None:
    """Element-wise parity that also covers non-finite and out-of-range results.

    Where the fp64 oracle gives NaN the GPU must give NaN; where it gives +-Inf, or a finite
    value beyond the output type's largest finite value by more than the tolerance, the GPU
    must give the infinity of the same sign; everywhere else the GPU value must be finite and
    within TOL * bound + floor of the oracle."""
    g = as_f64(gpu)
    rel = TOL[out_dtype]
    nan_ref = np.isnan(ref)
    big = np.isfinite(ref) & (np.abs(ref) > FINITE_MAX[out_dtype] + rel * np.abs(bound))
    inf_ref = np.isinf(ref) | big
    fin = ~nan_ref & ~inf_ref

    def first(mask, msg):
        if mask.any():
            i = int(np.flatnonzero(mask)[0])
            raise AssertionError(f"{what}: {int(mask.sum())} of {mask.size} elements {msg}; "
                                 f"first at {i}: gpu {g[i]!r} oracle {ref[i]!r} "
                                 f"bound {bound[i]!r}")

    first(nan_ref & ~np.isnan(g), "should be NaN")
    first(inf_ref & ~(np.isinf(g) & (np.sign(g) == np.sign(ref))), "should be an infinity of "
          "the oracle's sign")
    gf, rf, bf = g[fin], ref[fin], bound[fin]
    bad = np.zeros(ref.shape, dtype=bool)
    bad[fin] = ~(np.abs(gf - rf) <= rel * bf + floor)
    first(bad, "off")
