"""fp64 CPU oracle for the BaryCache skipped-step forecast (test infrastructure only).

Only ``tests/``, ``__graft_entry__.smoke()`` and the CPU-baseline leg of ``bench.py`` may
import this package.  The product library never calls it; it is the independent
reference the CUDA path is checked against.  The arithmetic lives in ``oracle.c``
(plain C, double precision); this module compiles it with gcc on first use and wraps the
entry points with ctypes and numpy.

Functions (paper: BaryCache, Sec. 3.2-3.3, Eqs. 8-13):

* :func:`lagrange` -- exact extrapolation coefficients, explicit Lagrange product.
* :func:`paper_weights` -- the stabilised weights of Eqs. 8-12.
* :func:`delta_table` -- the decay factor delta_H of Sec. 3.2.
* :func:`combine` -- Eq. 13 element by element, with the tolerance scale sum_j |W_j||F_j|.
* :func:`euler` -- Eq. 13 on the cached velocity followed by x + dt * v_hat.
* :func:`bf16_to_float64` -- exact widening of stored bf16 words.
* :func:`ddpm_coefficients` -- Eq. 3's mean and Eq. 2's deviation as x' = a x + b eps + c z.
* :func:`ddim_coefficients` -- the DDIM step (Song et al., ICLR 2021) in the same form.
* :func:`update` -- Eq. 13 on the cached model output, then x' = a x + b v_hat + c z.
* :func:`drift` -- the relative L1 probe drift of the adaptive schedule (Sec. 4.5).
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "oracle.c")
_LIB = os.path.join(_HERE, "liboracle.so")
_lock = threading.Lock()
_lib = None

OK, DUPLICATE_NODE, DEGENERATE, BAD_ARG = 0, 1, 2, 3
F32, BF16 = 0, 1


class OracleError(RuntimeError):
    pass


def build(force: bool = False) -> str:
    """Compile ``oracle.c`` into ``liboracle.so`` (gcc, -O2, no fast-math)."""
    if force or not os.path.exists(_LIB) or os.path.getmtime(_LIB) < os.path.getmtime(_SRC):
        tmp = _LIB + f".tmp{os.getpid()}"
        subprocess.check_call(
            ["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-fno-fast-math",
             "-ffp-contract=off", "-o", tmp, _SRC, "-lm"])
        os.replace(tmp, _LIB)
    return _LIB


def _load():
    global _lib
    with _lock:
        if _lib is None:
            # ORACLE_LIB points the pins at a deliberately broken build of oracle.c (the
            # mutation test); normally the oracle is built from its source here.
            path = os.environ.get("ORACLE_LIB") or build()
            lib = ctypes.CDLL(path)
            dp = ctypes.POINTER(ctypes.c_double)
            lib.oracle_lagrange.argtypes = [dp, ctypes.c_int, ctypes.c_double, dp]
            lib.oracle_lagrange.restype = ctypes.c_int
            lib.oracle_delta_table.argtypes = [ctypes.c_int]
            lib.oracle_delta_table.restype = ctypes.c_double
            lib.oracle_paper_weights.argtypes = [dp, ctypes.c_int, ctypes.c_double,
                                                 ctypes.c_double, ctypes.c_double,
                                                 ctypes.c_double, ctypes.c_double, dp]
            lib.oracle_paper_weights.restype = ctypes.c_int
            lib.oracle_bf16_to_double.argtypes = [ctypes.c_uint16]
            lib.oracle_bf16_to_double.restype = ctypes.c_double
            vpp = ctypes.POINTER(ctypes.c_void_p)
            lib.oracle_combine.argtypes = [ctypes.c_int, vpp, ctypes.c_int, dp,
                                           ctypes.c_int64, dp, dp]
            lib.oracle_combine.restype = None
            lib.oracle_euler.argtypes = [ctypes.c_int, vpp, ctypes.c_int, dp, ctypes.c_int64,
                                         ctypes.c_double, ctypes.c_int, ctypes.c_void_p,
                                         dp, dp, dp]
            lib.oracle_euler.restype = None
            d = ctypes.c_double
            lib.oracle_ddpm_coefficients.argtypes = [d, d, dp, dp, dp]
            lib.oracle_ddpm_coefficients.restype = ctypes.c_int
            lib.oracle_ddim_coefficients.argtypes = [d, d, d, dp, dp, dp]
            lib.oracle_ddim_coefficients.restype = ctypes.c_int
            lib.oracle_update.argtypes = [ctypes.c_int, vpp, ctypes.c_int, dp, ctypes.c_int64,
                                          d, d, d, ctypes.c_int, ctypes.c_void_p,
                                          ctypes.c_void_p, dp, dp]
            lib.oracle_update.restype = None
            lib.oracle_drift.argtypes = [ctypes.c_int, ctypes.c_void_p, ctypes.c_void_p,
                                         ctypes.c_int64, dp]
            lib.oracle_drift.restype = None
            _lib = lib
    return _lib


def _dptr(a: np.ndarray):
    return a.ctypes.data_as(ctypes.POINTER(ctypes.c_double))


def lagrange(nodes, t: float) -> np.ndarray:
    """Exact coefficients c_j = prod_{k!=j} (t-s_k)/(s_j-s_k); nodes newest first."""
    s = np.ascontiguousarray(nodes, dtype=np.float64)
    c = np.zeros(len(s), dtype=np.float64)
    rc = _load().oracle_lagrange(_dptr(s), len(s), float(t), _dptr(c))
    if rc != OK:
        raise OracleError(f"oracle_lagrange status {rc}")
    return c


def delta_table(H: int) -> float:
    """delta_H of Sec. 3.2: 1.0 (H=2), 0.95 (H=3), 0.7 (H=4); 1.0 for H=1."""
    d = _load().oracle_delta_table(int(H))
    if d <= 0:
        raise OracleError(f"no delta_H given for H={H}")
    return d


def paper_weights(nodes, t: float, delta: float | None = None, lam: float = 0.0,
                  C: float = 10.0, eta: float = 1e-12) -> np.ndarray:
    """Eqs. 8-12.  ``delta=None`` takes delta_H for H = len(nodes)."""
    s = np.ascontiguousarray(nodes, dtype=np.float64)
    if delta is None:
        delta = delta_table(len(s))
    W = np.zeros(len(s), dtype=np.float64)
    rc = _load().oracle_paper_weights(_dptr(s), len(s), float(t), float(delta), float(lam),
                                      float(C), float(eta), _dptr(W))
    if rc != OK:
        raise OracleError(f"oracle_paper_weights status {rc}")
    return W


def bf16_to_float64(bits) -> np.ndarray:
    """Widen bf16 words (uint16) to float64 through the oracle's own decoder."""
    b = np.asarray(bits, dtype=np.uint16)
    lib = _load()
    flat = b.reshape(-1)
    return np.array([lib.oracle_bf16_to_double(int(v)) for v in flat],
                    dtype=np.float64).reshape(b.shape)


def _dtype_code(a: np.ndarray) -> int:
    if a.dtype == np.float32:
        return F32
    if a.dtype == np.uint16:
        return BF16
    raise TypeError("stored tensors are float32 or bf16 bit patterns (uint16)")


def combine(F: list[np.ndarray], W) -> tuple[np.ndarray, np.ndarray]:
    """Eq. 13 over stored tensors F[j] (float32, or uint16 bf16 words), newest first.

    Returns (x_hat, bound) in float64, bound = sum_j |W_j| |F_j|.
    """
    W = np.ascontiguousarray(W, dtype=np.float64)
    m = len(W)
    if len(F) != m:
        raise ValueError("one stored tensor per weight")
    arrs = [np.ascontiguousarray(f).reshape(-1) for f in F]
    code = _dtype_code(arrs[0])
    n = arrs[0].size
    for a in arrs:
        if a.size != n or _dtype_code(a) != code:
            raise ValueError("stored tensors must share size and dtype")
    ptrs = (ctypes.c_void_p * m)(*[a.ctypes.data for a in arrs])
    out = np.empty(n, dtype=np.float64)
    bound = np.empty(n, dtype=np.float64)
    _load().oracle_combine(code, ptrs, m, _dptr(W), n, _dptr(out), _dptr(bound))
    return out, bound


def euler(V: list[np.ndarray], W, x: np.ndarray, dt: float):
    """Eq. 13 on the cached velocity, then x + dt * v_hat (explicit Euler).

    Returns (x_new, v_hat, bound), float64, bound = |x| + |dt| sum_j |W_j||V_j|.
    """
    W = np.ascontiguousarray(W, dtype=np.float64)
    m = len(W)
    arrs = [np.ascontiguousarray(v).reshape(-1) for v in V]
    code = _dtype_code(arrs[0])
    xa = np.ascontiguousarray(x).reshape(-1)
    n = arrs[0].size
    if xa.size != n:
        raise ValueError("x and the velocity must have the same size")
    ptrs = (ctypes.c_void_p * m)(*[a.ctypes.data for a in arrs])
    x_new = np.empty(n, dtype=np.float64)
    v_hat = np.empty(n, dtype=np.float64)
    bound = np.empty(n, dtype=np.float64)
    _load().oracle_euler(code, ptrs, m, _dptr(W), n, float(dt), _dtype_code(xa),
                         ctypes.c_void_p(xa.ctypes.data), _dptr(x_new), _dptr(v_hat),
                         _dptr(bound))
    return x_new, v_hat, bound


def ddpm_coefficients(alpha_t: float, alpha_bar_t: float) -> tuple[float, float, float]:
    a, b, c = ctypes.c_double(), ctypes.c_double(), ctypes.c_double()
    rc = _load().oracle_ddpm_coefficients(alpha_t, alpha_bar_t, ctypes.byref(a),
                                          ctypes.byref(b), ctypes.byref(c))
    if rc != OK:
        raise OracleError(f"oracle_ddpm_coefficients status {rc}")
    return a.value, b.value, c.value


def ddim_coefficients(alpha_bar_t: float, alpha_bar_prev: float,
                      eta: float = 0.0) -> tuple[float, float, float]:
    a, b, c = ctypes.c_double(), ctypes.c_double(), ctypes.c_double()
    rc = _load().oracle_ddim_coefficients(alpha_bar_t, alpha_bar_prev, eta, ctypes.byref(a),
                                          ctypes.byref(b), ctypes.byref(c))
    if rc != OK:
        raise OracleError(f"oracle_ddim_coefficients status {rc}")
    return a.value, b.value, c.value


def update(V: list[np.ndarray], W, x: np.ndarray, a: float, b: float, c: float = 0.0,
           z: np.ndarray | None = None):
    """Eq. 13 on the cached model output, then x' = a x + b v_hat + c z.

    Returns (x_new, bound), float64, bound = |a x| + |b| sum_j |W_j||V_j| + |c z|.
    """
    W = np.ascontiguousarray(W, dtype=np.float64)
    m = len(W)
    arrs = [np.ascontiguousarray(v).reshape(-1) for v in V]
    code = _dtype_code(arrs[0])
    xa = np.ascontiguousarray(x).reshape(-1)
    n = arrs[0].size
    za = None if z is None else np.ascontiguousarray(z).reshape(-1)
    if xa.size != n or (za is not None and (za.size != n or za.dtype != xa.dtype)):
        raise ValueError("x (and z) must match the velocity's size; z has x's dtype")
    ptrs = (ctypes.c_void_p * m)(*[v.ctypes.data for v in arrs])
    x_new = np.empty(n, dtype=np.float64)
    bound = np.empty(n, dtype=np.float64)
    _load().oracle_update(code, ptrs, m, _dptr(W), n, float(a), float(b), float(c),
                          _dtype_code(xa), ctypes.c_void_p(xa.ctypes.data),
                          None if za is None else ctypes.c_void_p(za.ctypes.data),
                          _dptr(x_new), _dptr(bound))
    return x_new, bound


def drift(cur: np.ndarray, prev: np.ndarray) -> np.ndarray:
    """[sum |cur - prev|, sum |prev|, ratio] in float64 (Sec. 4.5 probe drift)."""
    c = np.ascontiguousarray(cur).reshape(-1)
    p = np.ascontiguousarray(prev).reshape(-1)
    if c.size != p.size or c.dtype != p.dtype:
        raise ValueError("cur and prev must match")
    out = np.zeros(3, dtype=np.float64)
    _load().oracle_drift(_dtype_code(c), ctypes.c_void_p(c.ctypes.data),
                         ctypes.c_void_p(p.ctypes.data), c.size, _dptr(out))
    return out
