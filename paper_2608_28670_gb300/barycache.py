"""Thin ctypes binding of ``libbarycache.so`` (``include/barycache.h``).

Argument marshalling only: every function forwards to the C entry point of the same name
and raises :class:`BaryCacheError` on a non-OK status.  Device buffers are passed as
integer addresses (``tensor.data_ptr()``) and streams as integer handles
(``torch.cuda.current_stream().cuda_stream``); this module never touches device memory
itself and has no fallback: if the library is not built, the first call raises.
"""
from __future__ import annotations

import ctypes
import os
import threading
from typing import Sequence

import numpy as np

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "lib", "libbarycache.so")

BC_MAX_K = 4
OK, ERR_INVALID_ARG, ERR_ALIGNMENT, ERR_OOM, ERR_CUDA, ERR_NOT_READY, \
    ERR_DUPLICATE_NODE, ERR_DEGENERATE_WEIGHTS, ERR_BAD_HANDLE, ERR_DEVICE_TIMEOUT = range(10)
DTYPE_F32, DTYPE_BF16 = 0, 1
MODE_EXACT, MODE_PAPER = 0, 1
KERNEL_AUTO, KERNEL_REGISTER, KERNEL_PIPELINE = 0, 1, 2


class BaryCacheError(RuntimeError):
    def __init__(self, status: int, where: str, detail: str):
        super().__init__(f"{where}: status {status} ({detail})")
        self.status = status


class bc_params(ctypes.Structure):
    _fields_ = [("mode", ctypes.c_int32), ("delta", ctypes.c_double),
                ("lambda_", ctypes.c_double), ("clip_C", ctypes.c_double),
                ("eta", ctypes.c_double)]


class bc_adaptive(ctypes.Structure):
    _fields_ = [("threshold", ctypes.c_double), ("accumulated", ctypes.c_double),
                ("K", ctypes.c_int32), ("steps", ctypes.c_int32), ("full_steps", ctypes.c_int32)]


class bc_stats(ctypes.Structure):
    _fields_ = [("forecasts", ctypes.c_int64), ("pushes", ctypes.c_int64),
                ("kernel_launches", ctypes.c_int64), ("memo_hits", ctypes.c_int64),
                ("memo_misses", ctypes.c_int64), ("pipeline_launches", ctypes.c_int64),
                ("table_uploads", ctypes.c_int64)]


_lib = None
_lock = threading.Lock()

_SIGNATURES = {
    "bc_version": ([], ctypes.c_int),
    "bc_status_string": ([ctypes.c_int], ctypes.c_char_p),
    "bc_last_error": ([], ctypes.c_char_p),
    "bc_params_default": ([ctypes.POINTER(bc_params)], None),
    "bc_solve": ([ctypes.POINTER(ctypes.c_double), ctypes.c_int, ctypes.c_double,
                  ctypes.POINTER(bc_params), ctypes.POINTER(ctypes.c_double)], ctypes.c_int),
    "bc_cache_bytes_for": ([ctypes.POINTER(ctypes.c_int64), ctypes.c_int, ctypes.c_int,
                            ctypes.c_int, ctypes.POINTER(ctypes.c_int64)], ctypes.c_int),
    "bc_cache_create": ([ctypes.POINTER(ctypes.c_int64), ctypes.c_int, ctypes.c_int,
                         ctypes.c_int, ctypes.POINTER(bc_params),
                         ctypes.POINTER(ctypes.c_void_p)], ctypes.c_int),
    "bc_cache_destroy": ([ctypes.c_void_p], ctypes.c_int),
    "bc_cache_bytes": ([ctypes.c_void_p, ctypes.POINTER(ctypes.c_int64)], ctypes.c_int),
    "bc_cache_info": ([ctypes.c_void_p, ctypes.POINTER(ctypes.c_int), ctypes.POINTER(ctypes.c_int),
                       ctypes.POINTER(ctypes.c_int)], ctypes.c_int),
    "bc_cache_set_params": ([ctypes.c_void_p, ctypes.POINTER(bc_params)], ctypes.c_int),
    "bc_cache_reset": ([ctypes.c_void_p], ctypes.c_int),
    "bc_cache_push": ([ctypes.c_void_p, ctypes.POINTER(ctypes.c_void_p), ctypes.c_double,
                       ctypes.c_void_p], ctypes.c_int),
    "bc_cache_next_slot_ptrs": ([ctypes.c_void_p, ctypes.POINTER(ctypes.c_void_p)],
                                ctypes.c_int),
    "bc_cache_commit": ([ctypes.c_void_p, ctypes.c_double], ctypes.c_int),
    "bc_cache_nodes": ([ctypes.c_void_p, ctypes.POINTER(ctypes.c_double),
                        ctypes.POINTER(ctypes.c_int)], ctypes.c_int),
    "bc_cache_slot_ptrs": ([ctypes.c_void_p, ctypes.c_int, ctypes.POINTER(ctypes.c_void_p)],
                           ctypes.c_int),
    "bc_coefficients": ([ctypes.c_void_p, ctypes.c_double, ctypes.POINTER(ctypes.c_double),
                         ctypes.POINTER(ctypes.c_int)], ctypes.c_int),
    "bc_forecast": ([ctypes.c_void_p, ctypes.c_double, ctypes.POINTER(ctypes.c_void_p),
                     ctypes.c_int, ctypes.c_void_p], ctypes.c_int),
    "bc_forecast_step": ([ctypes.c_void_p, ctypes.c_double, ctypes.c_double,
                          ctypes.POINTER(ctypes.c_void_p), ctypes.c_int, ctypes.c_int,
                          ctypes.c_void_p, ctypes.c_int, ctypes.c_void_p], ctypes.c_int),
    "bc_cache_stats": ([ctypes.c_void_p, ctypes.POINTER(bc_stats)], ctypes.c_int),
    "bc_forecast_update": ([ctypes.c_void_p, ctypes.c_double, ctypes.c_double, ctypes.c_double,
                            ctypes.c_double, ctypes.POINTER(ctypes.c_void_p), ctypes.c_int,
                            ctypes.c_int, ctypes.c_void_p, ctypes.c_int, ctypes.c_void_p,
                            ctypes.c_void_p], ctypes.c_int),
    "bc_cache_push_flat": ([ctypes.c_void_p, ctypes.c_void_p, ctypes.c_double, ctypes.c_void_p],
                           ctypes.c_int),
    "bc_forecast_flat": ([ctypes.c_void_p, ctypes.c_double, ctypes.c_void_p, ctypes.c_void_p],
                         ctypes.c_int),
    "bc_cache_layout": ([ctypes.c_void_p, ctypes.POINTER(ctypes.c_int64)], ctypes.c_int),
    "bc_ddpm_coefficients": ([ctypes.c_double, ctypes.c_double, ctypes.POINTER(ctypes.c_double),
                              ctypes.POINTER(ctypes.c_double), ctypes.POINTER(ctypes.c_double)],
                             ctypes.c_int),
    "bc_ddim_coefficients": ([ctypes.c_double, ctypes.c_double, ctypes.c_double,
                              ctypes.POINTER(ctypes.c_double), ctypes.POINTER(ctypes.c_double),
                              ctypes.POINTER(ctypes.c_double)], ctypes.c_int),
    "bc_schedule_equal": ([ctypes.c_int, ctypes.c_int, ctypes.c_int,
                           ctypes.POINTER(ctypes.c_uint8)], ctypes.c_int),
    "bc_adaptive_init": ([ctypes.c_void_p, ctypes.c_double, ctypes.c_int], ctypes.c_int),
    "bc_adaptive_decide": ([ctypes.c_void_p, ctypes.c_double, ctypes.POINTER(ctypes.c_int)],
                           ctypes.c_int),
    "bc_probe_drift": ([ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p, ctypes.c_int64,
                        ctypes.c_int, ctypes.c_void_p, ctypes.c_void_p], ctypes.c_int),
    "bc_cache_check": ([ctypes.c_void_p], ctypes.c_int),
    "bc_cache_set_kernel": ([ctypes.c_void_p, ctypes.c_int], ctypes.c_int),
    "bc_cache_inject_fault": ([ctypes.c_void_p, ctypes.c_int], ctypes.c_int),
    "bc_probe_drift_noalloc": ([ctypes.c_void_p, ctypes.c_void_p, ctypes.c_int64, ctypes.c_int,
                                ctypes.c_void_p, ctypes.c_void_p], ctypes.c_int),
}


def exported_names() -> list[str]:
    return list(_SIGNATURES)


def lib() -> ctypes.CDLL:
    """Load the library (raises if it has not been built; there is no fallback)."""
    global _lib
    if _lib is not None:          # loaded: no lock on the per-call path
        return _lib
    with _lock:
        if _lib is None:
            if not os.path.exists(LIB_PATH):
                raise RuntimeError(
                    f"{LIB_PATH} is missing: build it with __graft_entry__.build() "
                    "(the forecast has no CPU fallback)")
            h = ctypes.CDLL(LIB_PATH)
            for name, (args, res) in _SIGNATURES.items():
                fn = getattr(h, name)
                fn.argtypes = args
                fn.restype = res
            _lib = h
    return _lib


def _check(status: int, where: str) -> None:
    if status != OK:
        L = lib()
        detail = L.bc_last_error().decode() or L.bc_status_string(status).decode()
        raise BaryCacheError(status, where, detail)


_PTR_ARRAY_TYPES: dict[int, type] = {}


def _ptr_array(ptrs):
    """A C array of device addresses.  A 1-D numpy array of uint64 / int64 addresses (0 for
    NULL) is passed without a copy when it is contiguous and writable (a ctypes array over
    its buffer, which keeps it alive for the call): for caches of thousands of tensors,
    converting a Python list element by element costs far more host time than the forecast
    itself, and numpy's ``ctypes.data_as`` alone costs several microseconds per call."""
    if isinstance(ptrs, np.ndarray):
        if ptrs.ndim != 1 or ptrs.dtype not in (np.uint64, np.int64):
            raise TypeError("pointer arrays must be 1-D uint64 or int64")
        arr_t = _PTR_ARRAY_TYPES.get(ptrs.size)
        if arr_t is None:
            arr_t = _PTR_ARRAY_TYPES.setdefault(ptrs.size, ctypes.c_void_p * ptrs.size)
        if ptrs.flags.c_contiguous and ptrs.flags.writeable:
            return arr_t.from_buffer(ptrs)
        return arr_t.from_buffer_copy(np.ascontiguousarray(ptrs))
    return (ctypes.c_void_p * len(ptrs))(*[p if p else None for p in ptrs])


# Layer counts of the handles this module created (dropped when it destroys them), so that a
# per-layer call does not pay an extra library round trip to learn the list length it must
# check.  Handles created elsewhere are asked every time.
_layer_counts: dict[int, int] = {}


def _layer_count(h: int) -> int:
    n = _layer_counts.get(h)
    if n is not None:
        return n
    c = ctypes.c_int()
    _check(lib().bc_cache_info(h, ctypes.byref(c), None, None), "bc_cache_info")
    return c.value


def _layer_ptrs(h: int, ptrs: Sequence[int | None], where: str):
    """Per-layer pointer array of exactly the cache's layer count (the C call reads that
    many entries, so a shorter list must never reach it)."""
    n = _layer_count(h)
    if len(ptrs) != n:
        raise BaryCacheError(ERR_INVALID_ARG, where,
                             f"{len(ptrs)} pointers given for a cache of {n} layers")
    return _ptr_array(ptrs)


def _params(mode=MODE_PAPER, delta=0.0, lam=0.0, clip_C=10.0, eta=1e-12) -> bc_params:
    return bc_params(mode, delta, lam, clip_C, eta)


def make_params(mode: int = MODE_PAPER, delta: float = 0.0, lam: float = 0.0,
                clip_C: float = 10.0, eta: float = 1e-12) -> bc_params:
    """Weight parameters (defaults are the paper's: PAPER mode, delta_H table, lambda 0,
    C 10, eta 1e-12)."""
    return _params(mode, delta, lam, clip_C, eta)


# ----------------------------------------------------------------------- host-only calls
def bc_version() -> int:
    return lib().bc_version()


def bc_params_default() -> bc_params:
    p = bc_params()
    lib().bc_params_default(ctypes.byref(p))
    return p


def bc_solve(nodes: Sequence[float], t: float, params: bc_params | None = None) -> list[float]:
    m = len(nodes)
    arr = (ctypes.c_double * max(m, 1))(*nodes)
    out = (ctypes.c_double * max(m, 1))()
    _check(lib().bc_solve(arr, m, float(t), ctypes.byref(params) if params else None, out),
           "bc_solve")
    return list(out[:m])


def bc_cache_bytes_for(numels: Sequence[int], K: int, dtype: int) -> int:
    arr = (ctypes.c_int64 * len(numels))(*numels)
    out = ctypes.c_int64()
    _check(lib().bc_cache_bytes_for(arr, len(numels), K, dtype, ctypes.byref(out)),
           "bc_cache_bytes_for")
    return out.value


# ----------------------------------------------------------------------- handle calls
def bc_cache_create(numels: Sequence[int], K: int, dtype: int,
                    params: bc_params | None = None) -> int:
    arr = (ctypes.c_int64 * len(numels))(*numels)
    h = ctypes.c_void_p()
    _check(lib().bc_cache_create(arr, len(numels), K, dtype,
                                 ctypes.byref(params) if params else None, ctypes.byref(h)),
           "bc_cache_create")
    _layer_counts[h.value] = len(numels)
    return h.value


def bc_cache_destroy(h: int) -> None:
    _layer_counts.pop(h, None)
    _check(lib().bc_cache_destroy(h), "bc_cache_destroy")


def bc_cache_bytes(h: int) -> int:
    out = ctypes.c_int64()
    _check(lib().bc_cache_bytes(h, ctypes.byref(out)), "bc_cache_bytes")
    return out.value


def bc_cache_set_params(h: int, params: bc_params) -> None:
    _check(lib().bc_cache_set_params(h, ctypes.byref(params)), "bc_cache_set_params")


def bc_cache_reset(h: int) -> None:
    _check(lib().bc_cache_reset(h), "bc_cache_reset")


def bc_cache_info(h: int) -> tuple[int, int, int]:
    """(n_layers, K, dtype) of a cache."""
    n, k, d = ctypes.c_int(), ctypes.c_int(), ctypes.c_int()
    _check(lib().bc_cache_info(h, ctypes.byref(n), ctypes.byref(k), ctypes.byref(d)),
           "bc_cache_info")
    return n.value, k.value, d.value


def bc_cache_push(h: int, layer_ptrs: Sequence[int], t: float, stream: int = 0) -> None:
    _check(lib().bc_cache_push(h, _layer_ptrs(h, layer_ptrs, "bc_cache_push"), float(t),
                               stream or None), "bc_cache_push")


def bc_cache_push_flat(h: int, src: int, t: float, stream: int = 0) -> None:
    _check(lib().bc_cache_push_flat(h, src or None, float(t), stream or None),
           "bc_cache_push_flat")


def bc_cache_next_slot_ptrs(h: int, n_layers: int | None = None) -> list[int]:
    n_layers = _layer_count(h)        # the array the C call fills has exactly this size
    out = (ctypes.c_void_p * n_layers)()
    _check(lib().bc_cache_next_slot_ptrs(h, out), "bc_cache_next_slot_ptrs")
    return [v or 0 for v in out]


def bc_cache_commit(h: int, t: float) -> None:
    _check(lib().bc_cache_commit(h, float(t)), "bc_cache_commit")


def bc_cache_nodes(h: int) -> list[float]:
    out = (ctypes.c_double * BC_MAX_K)()
    m = ctypes.c_int()
    _check(lib().bc_cache_nodes(h, out, ctypes.byref(m)), "bc_cache_nodes")
    return list(out[:m.value])


def bc_cache_slot_ptrs(h: int, j: int, n_layers: int | None = None) -> list[int]:
    n_layers = _layer_count(h)
    out = (ctypes.c_void_p * n_layers)()
    _check(lib().bc_cache_slot_ptrs(h, j, out), "bc_cache_slot_ptrs")
    return [v or 0 for v in out]


def bc_coefficients(h: int, t_new: float) -> list[float]:
    out = (ctypes.c_double * BC_MAX_K)()
    m = ctypes.c_int()
    _check(lib().bc_coefficients(h, float(t_new), out, ctypes.byref(m)), "bc_coefficients")
    return list(out[:m.value])


def bc_forecast(h: int, t_new: float, out_ptrs: Sequence[int | None], out_dtype: int,
                stream: int = 0) -> None:
    _check(lib().bc_forecast(h, float(t_new), _layer_ptrs(h, out_ptrs, "bc_forecast"), out_dtype,
                             stream or None), "bc_forecast")


def bc_forecast_step(h: int, t_new: float, dt: float, out_ptrs: Sequence[int | None],
                     out_dtype: int, v_layer: int, x: int, x_dtype: int,
                     stream: int = 0) -> None:
    _check(lib().bc_forecast_step(h, float(t_new), float(dt),
                                  _layer_ptrs(h, out_ptrs, "bc_forecast_step"), out_dtype,
                                  v_layer, x or None, x_dtype, stream or None),
           "bc_forecast_step")


def bc_cache_stats(h: int) -> dict:
    s = bc_stats()
    _check(lib().bc_cache_stats(h, ctypes.byref(s)), "bc_cache_stats")
    return {k: getattr(s, k) for k, _ in bc_stats._fields_}


def bc_forecast_update(h: int, t_new: float, a: float, b: float, c: float,
                       out_ptrs: Sequence[int | None], out_dtype: int, v_layer: int, x: int,
                       x_dtype: int, z: int | None = None, stream: int = 0) -> None:
    _check(lib().bc_forecast_update(h, float(t_new), float(a), float(b), float(c),
                                    _layer_ptrs(h, out_ptrs, "bc_forecast_update"), out_dtype,
                                    v_layer, x or None,
                                    x_dtype, z or None, stream or None), "bc_forecast_update")


def bc_forecast_flat(h: int, t_new: float, out: int, stream: int = 0) -> None:
    _check(lib().bc_forecast_flat(h, float(t_new), out or None, stream or None),
           "bc_forecast_flat")


def bc_cache_layout(h: int, n_layers: int | None = None) -> list[int]:
    n_layers = _layer_count(h)
    out = (ctypes.c_int64 * (n_layers + 1))()
    _check(lib().bc_cache_layout(h, out), "bc_cache_layout")
    return list(out)


def bc_ddpm_coefficients(alpha_t: float, alpha_bar_t: float) -> tuple[float, float, float]:
    a, b, c = ctypes.c_double(), ctypes.c_double(), ctypes.c_double()
    _check(lib().bc_ddpm_coefficients(float(alpha_t), float(alpha_bar_t), ctypes.byref(a),
                                      ctypes.byref(b), ctypes.byref(c)), "bc_ddpm_coefficients")
    return a.value, b.value, c.value


def bc_ddim_coefficients(alpha_bar_t: float, alpha_bar_prev: float,
                         eta: float = 0.0) -> tuple[float, float, float]:
    a, b, c = ctypes.c_double(), ctypes.c_double(), ctypes.c_double()
    _check(lib().bc_ddim_coefficients(float(alpha_bar_t), float(alpha_bar_prev), float(eta),
                                      ctypes.byref(a), ctypes.byref(b), ctypes.byref(c)),
           "bc_ddim_coefficients")
    return a.value, b.value, c.value


def bc_schedule_equal(n_steps: int, interval: int, K: int) -> list[int]:
    out = (ctypes.c_uint8 * max(n_steps, 1))()
    _check(lib().bc_schedule_equal(n_steps, interval, K, out), "bc_schedule_equal")
    return list(out[:n_steps])


def bc_adaptive_init(threshold: float, K: int) -> bc_adaptive:
    st = bc_adaptive()
    _check(lib().bc_adaptive_init(ctypes.byref(st), float(threshold), K), "bc_adaptive_init")
    return st


def bc_adaptive_decide(st: bc_adaptive, drift: float) -> int:
    full = ctypes.c_int()
    _check(lib().bc_adaptive_decide(ctypes.byref(st), float(drift), ctypes.byref(full)),
           "bc_adaptive_decide")
    return full.value


def bc_probe_drift(h: int, cur: int, prev: int, n: int, dtype: int, out: int,
                   stream: int = 0) -> None:
    _check(lib().bc_probe_drift(h, cur or None, prev or None, n, dtype, out or None,
                                stream or None), "bc_probe_drift")


def bc_probe_drift_noalloc(cur: int, prev: int, n: int, dtype: int, out: int,
                           stream: int = 0) -> None:
    """bc_probe_drift without a handle or any device allocation (static library scratch)."""
    _check(lib().bc_probe_drift_noalloc(cur or None, prev or None, n, dtype, out or None,
                                        stream or None), "bc_probe_drift_noalloc")


def bc_cache_check(h: int) -> None:
    """Raise BaryCacheError(ERR_DEVICE_TIMEOUT) if a forecast launch gave up waiting."""
    _check(lib().bc_cache_check(h), "bc_cache_check")


def bc_cache_inject_fault(h: int, what: int = 1) -> None:
    """Test hook: make the next forecast launch's pipeline wait run out (what = 1)."""
    _check(lib().bc_cache_inject_fault(h, what), "bc_cache_inject_fault")


def bc_cache_set_kernel(h: int, kernel: int) -> None:
    """Pin the forecast kernel (KERNEL_AUTO, KERNEL_REGISTER or KERNEL_PIPELINE)."""
    _check(lib().bc_cache_set_kernel(h, kernel), "bc_cache_set_kernel")
