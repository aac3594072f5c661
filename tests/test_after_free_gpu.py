"""HBM bandwidth right after freeing a very large allocation.

Freeing a large device allocation costs HBM bandwidth for a short while afterwards.  On GB300,
after freeing a 170 GB cache a new cache's forecasts stream at about 5.0 instead of 7.1 TB/s
for about 70 ms and then at full speed.  It does not matter whether the freed memory was ever
written, whether the library or torch freed it, whether a small allocation comes in between,
or where the new cache is placed (the same address as a later full-speed one).  After freeing
40 GB there is no visible dip.  So it is a transient of the driver's work on freed memory, not
a placement effect of bc_cache_create, and bench.py warms every leg up for at least 0.25 s.

This test frees a 120 GB cache, creates a c2i-512-shaped cache right away (K = 4, 2.6 GB moved
per forecast) and times forecasts in groups of ten for 0.5 s: from 0.25 s after the free on,
every group must run within 10 % of the settled rate.
"""
import statistics
import time

import pytest
import torch

from paper_2608_28670_gb300 import barycache as bc
from paper_2608_28670_gb300.configs import WORKLOADS
from paper_2608_28670_gb300.runner import WorkloadRun

pytestmark = pytest.mark.gpu

BIG_BYTES = 120 * 10**9
RECOVERED_BY_S = 0.25


def test_bandwidth_recovers_soon_after_a_large_free():
    torch.cuda.set_device(0)
    torch.cuda.empty_cache()
    free, _ = torch.cuda.mem_get_info()
    if free < BIG_BYTES + 8 * 10**9:
        pytest.skip(f"needs {BIG_BYTES / 1e9:.0f} GB free on the device, {free / 1e9:.0f} GB is")
    n = BIG_BYTES // 2 // 60
    big = bc.bc_cache_create([n] * 60, 1, bc.DTYPE_BF16)
    bc.bc_cache_destroy(big)
    t_free = time.perf_counter()
    stream = torch.cuda.current_stream().cuda_stream
    r = WorkloadRun(WORKLOADS["c2i-512"], stream=stream)
    try:
        samples = []
        while time.perf_counter() - t_free < 0.5:
            a = torch.cuda.Event(enable_timing=True)
            b = torch.cuda.Event(enable_timing=True)
            a.record()
            for _ in range(10):
                r.forecast()
            b.record()
            torch.cuda.synchronize()
            ms = a.elapsed_time(b) / 10
            samples.append((time.perf_counter() - t_free, r.algorithmic_bytes() / (ms * 1e-3) / 1e9))
        bc.bc_cache_check(r.h)
    finally:
        r.close()
    settled = statistics.median(g for t, g in samples if t > 0.35)
    late = [(t, g) for t, g in samples if t > RECOVERED_BY_S]
    assert late and settled > 0
    slow = [(round(t, 3), round(g)) for t, g in late if g < 0.9 * settled]
    dip = [t for t, g in samples if g < 0.9 * settled]
    print(f"settled {settled:.0f} GB/s; below 90 % until {max(dip) if dip else 0.0:.3f} s "
          f"after the free; first group {samples[0][1]:.0f} GB/s at {samples[0][0]:.3f} s")
    assert not slow, f"still below 90 % of {settled:.0f} GB/s after {RECOVERED_BY_S} s: {slow[:5]}"
