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
