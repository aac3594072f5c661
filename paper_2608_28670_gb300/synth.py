"""Seeded synthetic inputs for the forecast (shared by tests and the benchmark).

Holds none of the forecast's arithmetic: it only produces feature tensors.  Two sources:

* host (numpy) trajectories for small parity cases -- :func:`host_trajectories`;
* the device generator ``libbc_synth.so`` (Philox4x32-10 + Box-Muller) for full-size
  workloads -- :func:`fill_device`.  Its output depends only on (seed, tensor id, step id,
  element index), so a benchmark can write history slots in place without host copies.

Feature recipe (both sources): each element follows a random polynomial of degree `degree`
in the normalised time tau with N(0, 1) coefficients, times an outlier amplitude on a
seeded fraction of channels, plus N(0, noise_std^2) noise drawn per step.
"""
from __future__ import annotations

import ctypes
import os
import threading

import numpy as np

_PKG = os.path.dirname(os.path.abspath(__file__))
SYNTH_LIB = os.path.join(_PKG, "lib", "libbc_synth.so")

_lib = None
_lock = threading.Lock()


def f32_to_bf16_bits(a: np.ndarray) -> np.ndarray:
    """Round float32 to bf16 (nearest, ties to even) and return the uint16 bit patterns."""
    b = np.ascontiguousarray(a, dtype=np.float32).view(np.uint32).astype(np.uint64)
    rounded = (b + 0x7FFF + ((b >> 16) & 1)) >> 16
    return rounded.astype(np.uint16)


def bf16_bits_to_f32(bits: np.ndarray) -> np.ndarray:
    return (np.asarray(bits, dtype=np.uint16).astype(np.uint32) << 16).view(np.float32)


def host_trajectories(shapes, taus, *, dtype: str, degree: int = 2, noise_std: float = 1e-3,
                      hidden: int | None = None, outlier_frac: float = 0.0,
                      outlier_scale: float = 10.0, seed: int = 2026):
    """Features of every layer at every normalised time in `taus`.

    Returns ``feats[i][l]``: layer l at time taus[i], as float32 (dtype "f32") or as bf16
    bit patterns in uint16 (dtype "bf16"), shaped like ``shapes[l]``.
    """
    rng = np.random.default_rng(seed)
    coefs, amps = [], []
    for shp in shapes:
        n = int(np.prod(shp))
        coefs.append(rng.standard_normal((degree + 1, n)))
        amp = np.ones(n)
        if outlier_frac > 0 and n > 0:
            h = hidden or shp[-1]
            ch = rng.random(h) < outlier_frac
            amp = np.where(ch[np.arange(n) % h], outlier_scale, 1.0)
        amps.append(amp)
    feats = []
    for tau in taus:
        per_layer = []
        for shp, c, amp in zip(shapes, coefs, amps):
            v = np.polynomial.polynomial.polyval(tau, c) * amp
            v = v + noise_std * rng.standard_normal(v.shape)
            v = v.astype(np.float32).reshape(shp)
            per_layer.append(f32_to_bf16_bits(v) if dtype == "bf16" else v)
        feats.append(per_layer)
    return feats


def _load():
    global _lib
    with _lock:
        if _lib is None:
            if not os.path.exists(SYNTH_LIB):
                raise RuntimeError(f"{SYNTH_LIB} is missing: run __graft_entry__.build()")
            L = ctypes.CDLL(SYNTH_LIB)
            L.bcs_fill.argtypes = [ctypes.c_void_p, ctypes.c_int, ctypes.c_int64,
                                   ctypes.c_uint64, ctypes.c_uint32, ctypes.c_uint32,
                                   ctypes.c_double, ctypes.c_int, ctypes.c_double,
                                   ctypes.c_int64, ctypes.c_double, ctypes.c_double,
                                   ctypes.c_void_p]
            L.bcs_fill.restype = ctypes.c_int
            _lib = L
    return _lib


def fill_device(ptr: int, dtype: int, n: int, *, seed: int, tensor_id: int, step_id: int,
                tau: float, degree: int, noise_std: float, hidden: int = 1,
                outlier_frac: float = 0.0, outlier_scale: float = 10.0, stream: int = 0):
    """Write n trajectory values (dtype 0 = f32, 1 = bf16) at device address `ptr`."""
    rc = _load().bcs_fill(ptr or None, dtype, n, seed, tensor_id, step_id, tau, degree,
                          noise_std, hidden, outlier_frac, outlier_scale, stream or None)
    if rc != 0:
        raise RuntimeError(f"bcs_fill failed with CUDA error {rc}")
