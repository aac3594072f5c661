"""Drive one workload through the C ABI: cache, in-place history, outputs, forecasts.

Used by the benchmark and by the full-size tests.  The K history slots are written in
place (zero-copy push: ``bc_cache_next_slot_ptrs`` + ``bc_cache_commit``) by the seeded
device generator, oldest node first, exactly as a DiT would write its block outputs on
full steps.  Output buffers are torch allocations; when a workload's cache plus a
full-size output would exceed its stated device-memory budget, the forecast is issued
over windows of layers (NULL outputs elsewhere), reusing one window of output buffers.
"""
from __future__ import annotations

import numpy as np
import torch

from . import barycache as bc
from . import synth
from .configs import Workload

SEED = 2026


class _CudaArray:
    def __init__(self, ptr: int, n: int, typestr: str):
        self.__cuda_array_interface__ = {"shape": (n,), "typestr": typestr,
                                         "data": (ptr, False), "version": 3, "strides": None}


def device_view(ptr: int, n: int, dtype: int) -> torch.Tensor:
    """Zero-copy 1-D torch view of `n` elements at device address `ptr` (bf16 as int16)."""
    typestr = "<f4" if dtype == bc.DTYPE_F32 else "<i2"
    return torch.as_tensor(_CudaArray(ptr, n, typestr), device="cuda")


class WorkloadRun:
    def __init__(self, w: Workload, K: int | None = None, out_dtype: int | None = None,
                 budget_bytes: int | None = None, params=None, seed: int = SEED,
                 stream: int = 0):
        self.w = w
        self.K = K or w.K
        self.seed = seed
        self.stream = stream
        self.out_dtype = w.dtype if out_dtype is None else out_dtype
        self.problem = w.representative(self.K)
        self.numels = w.numels
        self.n_feat = w.n_layers                # block outputs (the Euler layer follows)
        self.euler = w.euler_shape is not None
        self.h = bc.bc_cache_create(self.numels, self.K, w.dtype, params)
        try:
            self._fill_history()
            out_eb = 2 if self.out_dtype == bc.DTYPE_BF16 else 4
            layer_out = w.layer_numel * out_eb
            cache = bc.bc_cache_bytes(self.h)
            window = self.n_feat
            if budget_bytes is not None and cache + self.n_feat * layer_out > budget_bytes:
                window = max(1, (budget_bytes - cache) // layer_out)
                window = min(window, self.n_feat)
            self.window = int(window)
            self.calls = -(-self.n_feat // self.window)
            tdt = torch.float32 if self.out_dtype == bc.DTYPE_F32 else torch.bfloat16
            # one buffer, each window layer's output at a 256-byte aligned offset, so that
            # consecutive outputs can also be moved as one span
            stride = -(-w.layer_numel * out_eb // 256) * 256 // out_eb
            self._out_flat = torch.empty(stride * self.window, dtype=tdt, device="cuda")
            self.outs = [self._out_flat[i * stride:i * stride + w.layer_numel]
                         for i in range(self.window)]
            # per-call output tables, built once (the binding passes numpy tables as is)
            self._call_ptrs = [np.array([q or 0 for q in self.out_ptrs(c)], dtype=np.uint64)
                               for c in range(self.calls)]
            self.x = None
            if self.euler:
                nx = self.numels[-1]
                self.x = torch.empty(nx, dtype=torch.float32, device="cuda")
                self.reset_x()
        except Exception:
            bc.bc_cache_destroy(self.h)
            raise

    # ------------------------------------------------------------------ setup
    def _fill_history(self):
        p = self.problem
        steps = p.node_steps or tuple(range(len(p.nodes) - 1, -1, -1))
        for step, t in reversed(list(zip(steps, p.nodes))):   # oldest first
            ptrs = bc.bc_cache_next_slot_ptrs(self.h, len(self.numels))
            for l, n in enumerate(self.numels):
                synth.fill_device(ptrs[l], self.w.dtype, n, seed=self.seed, tensor_id=l,
                                  step_id=step, tau=self.w.tau(t), degree=self.w.degree,
                                  noise_std=self.w.noise_std, hidden=self.w.hidden,
                                  outlier_frac=self.w.outlier_frac,
                                  outlier_scale=self.w.outlier_scale, stream=self.stream)
            bc.bc_cache_commit(self.h, t)

    def reset_x(self):
        synth.fill_device(self.x.data_ptr(), bc.DTYPE_F32, self.x.numel(), seed=self.seed + 1,
                          tensor_id=0, step_id=0, tau=0.0, degree=0, noise_std=0.0,
                          stream=self.stream)

    # ------------------------------------------------------------------ the hot path
    def out_ptrs(self, call: int) -> list[int | None]:
        ptrs: list[int | None] = [None] * len(self.numels)
        lo = call * self.window
        for i in range(self.window):
            if lo + i < self.n_feat:
                ptrs[lo + i] = self.outs[i].data_ptr()
        return ptrs

    def forecast_call(self, call: int, t: float | None = None) -> None:
        """One C-ABI call: the forecast of one window of layers (plus, on the first
        window, the fused Euler step on the velocity layer)."""
        t = self.problem.t if t is None else t
        ptrs = self._call_ptrs[call]
        if self.euler and call == 0:
            bc.bc_forecast_step(self.h, t, self.problem.dt, ptrs, self.out_dtype,
                                len(self.numels) - 1, self.x.data_ptr(), bc.DTYPE_F32,
                                self.stream)
        else:
            bc.bc_forecast(self.h, t, ptrs, self.out_dtype, self.stream)

    def forecast(self, t: float | None = None) -> None:
        """One skipped step: every cached layer forecast once."""
        for c in range(self.calls):
            self.forecast_call(c, t)

    # ------------------------------------------------------------------ accounting
    def algorithmic_bytes(self) -> int:
        """HBM bytes one skipped step must move: K history reads + one output write per
        element, plus the Euler state read and write."""
        eb = self.w.elem_bytes
        ob = 2 if self.out_dtype == bc.DTYPE_BF16 else 4
        b = (self.K * eb + ob) * self.w.layer_numel * self.n_feat
        if self.euler:
            b += (self.K * eb + 2 * 4) * self.numels[-1]
        return b

    def elements(self) -> int:
        return sum(self.numels)

    def stats(self) -> dict:
        return bc.bc_cache_stats(self.h)

    def close(self):
        if self.h:
            bc.bc_cache_destroy(self.h)
            self.h = 0
        self.outs = []
        self._out_flat = None
        self.x = None
