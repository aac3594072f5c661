"""Several host threads driving the library at once.

The ABI allows one handle per thread; the library's own shared state (the handle registry,
per-device SM counts, occupancies and kernel attributes, the thread-local error message)
must stand up to concurrent calls.  Four threads, each with its own handle, stream, layer
shapes, history length and kernel choice, push, forecast and probe concurrently while a
fifth creates and destroys handles in a loop; every thread's outputs are then checked
against the oracle.  The first calls of every launch path happen inside the threads, so
the first-use caches are filled concurrently.
"""
import threading

import numpy as np
import pytest
import torch

import oracle
from paper_2608_28670_gb300 import barycache as bc
from paper_2608_28670_gb300 import synth
from tests.gpu_helpers import assert_close, oracle_weights, to_device, to_host

pytestmark = pytest.mark.gpu

CASES = [  # (numels, K, dtype, kernel)
    ([40_000_000 + 3], 3, bc.DTYPE_BF16, bc.KERNEL_AUTO),        # pipeline paths under AUTO
    ([100_003, 8192, 5], 2, bc.DTYPE_F32, bc.KERNEL_REGISTER),
    ([3 * 8192 + 1] * 12, 3, bc.DTYPE_BF16, bc.KERNEL_PIPELINE),
    ([65_536] * 70, 4, bc.DTYPE_BF16, bc.KERNEL_AUTO),           # 64+ layers: large table
]
TIMES = [0.9, 0.85, 0.8, 0.75]
ROUNDS = 15


def worker(idx, case, feats, out, errors, start):
    numels, K, dt, kernel = case
    try:
        torch.cuda.set_device(0)
        s = torch.cuda.Stream()
        start.wait(timeout=300)
        h = bc.bc_cache_create(numels, K, dt)
        try:
            bc.bc_cache_set_kernel(h, kernel)
            with torch.cuda.stream(s):
                for t, per in zip(TIMES[:K], feats):
                    dev = [to_device(f) for f in per]
                    bc.bc_cache_push(h, [d.data_ptr() for d in dev], t, s.cuda_stream)
                    s.synchronize()
                outs = [torch.empty(n, dtype=torch.float32 if dt == bc.DTYPE_F32
                                    else torch.int16, device="cuda") for n in numels]
                drift = torch.empty(3, dtype=torch.float64, device="cuda")
                for _ in range(ROUNDS):
                    bc.bc_forecast(h, 0.7, np.array([o.data_ptr() for o in outs], np.uint64),
                                   dt, s.cuda_stream)
                    slots = [bc.bc_cache_slot_ptrs(h, j, len(numels))[0] for j in range(2)]
                    bc.bc_probe_drift(h, slots[0], slots[1], numels[0], dt, drift.data_ptr(),
                                      s.cuda_stream)
                s.synchronize()
                bc.bc_cache_check(h)
                out[idx] = ([to_host(o, dt) for o in outs], drift.cpu().numpy())
        finally:
            bc.bc_cache_destroy(h)
    except Exception as e:  # reported by the main thread
        errors[idx] = e


def churn(stop, errors):
    try:
        torch.cuda.set_device(0)
        while not stop.is_set():
            h = bc.bc_cache_create([1024, 7], 2, bc.DTYPE_BF16)
            assert bc.bc_cache_info(h) == (2, 2, bc.DTYPE_BF16)
            bc.bc_cache_destroy(h)
    except Exception as e:
        errors["churn"] = e


def test_concurrent_handles_on_their_own_streams():
    import __graft_entry__
    __graft_entry__.build_libraries()
    torch.cuda.set_device(0)
    feats = [synth.host_trajectories([(n,) for n in numels], TIMES[:K],
                                     dtype="f32" if dt == bc.DTYPE_F32 else "bf16", seed=50 + i)
             for i, (numels, K, dt, _) in enumerate(CASES)]
    out, errors = {}, {}
    start, stop = threading.Barrier(len(CASES)), threading.Event()
    ch = threading.Thread(target=churn, args=(stop, errors))
    ch.start()
    threads = [threading.Thread(target=worker, args=(i, c, feats[i], out, errors, start))
               for i, c in enumerate(CASES)]
    for t in threads:
        t.start()
    for t in threads:
        t.join()
    stop.set()
    ch.join()
    assert not errors, errors
    rng = np.random.default_rng(0)
    for i, (numels, K, dt, _) in enumerate(CASES):
        got, drift = out[i]
        nodes = TIMES[:K][::-1]
        W = oracle_weights(nodes, 0.7, bc.MODE_PAPER)
        newest_first = feats[i][::-1]
        for l, n in enumerate(numels):
            idx = np.arange(n) if n <= 200_000 else np.unique(rng.integers(0, n, 20_000))
            ref, bound = oracle.combine([f[l].reshape(-1)[idx] for f in newest_first], W)
            assert_close(got[l][idx], ref, bound, dt, f"thread {i} layer {l}")
        ref_d = oracle.drift(newest_first[0][0].reshape(-1), newest_first[1][0].reshape(-1))
        np.testing.assert_allclose(drift, ref_d, rtol=2e-6)
