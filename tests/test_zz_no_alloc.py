"""The no-allocation probe drift (bc_probe_drift_noalloc).

Some callers cannot call cudaMalloc, nor let a library allocate for them: code inside a host
framework that owns all device memory, or a latency-bound loop that cannot take the implicit
device synchronisation of an allocation.  For them the library offers the probe drift with its
reduction scratch in the library's own static device memory.  These tests call it through the
C ABI and check it against the fp64 oracle and against the handle-based bc_probe_drift, on two
calls in a row, with the tolerance the drift tests use, from an empty probe up to exactly the
largest probe the static scratch holds (1 GiB per tensor).  The file is named to be collected
last.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2608_28670_gb300 import barycache as bc
from paper_2608_28670_gb300 import synth

RTOL = 2e-6          # the tolerance of the drift parity tests
MAX_ELEMS = {bc.DTYPE_BF16: 1 << 29, bc.DTYPE_F32: 1 << 28}   # 1 GiB per tensor


@pytest.fixture(scope="module")
def built():
    import __graft_entry__
    __graft_entry__.build_libraries()


def _inputs(n, dt, seed):
    """Host (stored) and device copies of a probe pair: prev, and cur = prev plus a change."""
    rng = np.random.default_rng(seed)
    if n > (1 << 26):
        # large probes: draw bf16 / fp32 bit patterns directly (values of magnitude 2^-8 .. 2^8
        # with random signs), which is much faster than normal deviates at this size
        if dt == bc.DTYPE_BF16:
            prev = rng.integers(0x3B80, 0x4380, n, dtype=np.uint16)
            prev |= (rng.integers(0, 2, n, dtype=np.uint16) << 15)
            cur = prev ^ rng.integers(0, 8, n, dtype=np.uint16)        # low mantissa bits
            dev = (torch.from_numpy(cur.view(np.int16)).cuda(),
                   torch.from_numpy(prev.view(np.int16)).cuda())
        else:
            pb = rng.integers(0x3B800000, 0x43800000, n, dtype=np.uint32)
            pb |= (rng.integers(0, 2, n, dtype=np.uint32) << 31)
            cb = pb ^ rng.integers(0, 1 << 16, n, dtype=np.uint32)
            prev, cur = pb.view(np.float32), cb.view(np.float32)
            dev = torch.from_numpy(cur).cuda(), torch.from_numpy(prev).cuda()
        return cur, prev, dev
    prev = rng.standard_normal(n).astype(np.float32)
    cur = prev + 0.05 * rng.standard_normal(n).astype(np.float32)
    if dt == bc.DTYPE_BF16:
        prev, cur = synth.f32_to_bf16_bits(prev), synth.f32_to_bf16_bits(cur)
        return cur, prev, (torch.from_numpy(cur.view(np.int16)).cuda(),
                           torch.from_numpy(prev.view(np.int16)).cuda())
    return cur, prev, (torch.from_numpy(cur).cuda(), torch.from_numpy(prev).cuda())


def _check(dt, n, seed):
    torch.cuda.set_device(0)
    cur_h, prev_h, (cur, prev) = _inputs(n, dt, seed)
    s = torch.cuda.current_stream().cuda_stream
    h = bc.bc_cache_create([16], 2, bc.DTYPE_BF16)
    try:
        ref = torch.empty(3, dtype=torch.float64, device="cuda")
        bc.bc_probe_drift(h, cur.data_ptr(), prev.data_ptr(), n, dt, ref.data_ptr(), s)
        outs = torch.full((2, 3), -1.0, dtype=torch.float64, device="cuda")
        for k in range(2):       # two calls in a row share the static scratch
            bc.bc_probe_drift_noalloc(cur.data_ptr(), prev.data_ptr(), n, dt,
                                      outs[k].data_ptr(), s)
        torch.cuda.synchronize()
        r = ref.cpu().numpy()
        o = outs.cpu().numpy()
        assert np.array_equal(o[0], o[1])
        exact = oracle.drift(cur_h, prev_h)
        for k in range(2):
            if n == 0:
                assert list(o[k]) == [0.0, 0.0, 0.0]
            else:
                np.testing.assert_allclose(o[k], exact, rtol=RTOL, atol=0.0)
            np.testing.assert_allclose(o[k], r, rtol=RTOL, atol=0.0)
    finally:
        bc.bc_cache_destroy(h)


@pytest.mark.gpu
@pytest.mark.parametrize("dt", [bc.DTYPE_BF16, bc.DTYPE_F32])
@pytest.mark.parametrize("n", [0, 5, 8, 4099, 1_048_576 + 9, 40_000_000 + 3])
def test_no_alloc_drift_matches_oracle_and_handle_drift_twice(built, dt, n):
    _check(dt, n, seed=n + 7 * dt)


@pytest.mark.gpu
@pytest.mark.parametrize("dt", [bc.DTYPE_BF16, bc.DTYPE_F32])
def test_no_alloc_drift_at_its_maximum_size(built, dt):
    # exactly the largest probe the static scratch holds (every one of its tiles is used)
    _check(dt, MAX_ELEMS[dt], seed=3 + dt)


def test_no_alloc_drift_rejects_sizes_beyond_its_scratch(built):
    # The size check happens on the host before any device work, so no GPU is needed.
    for dt, n_max in MAX_ELEMS.items():
        with pytest.raises(bc.BaryCacheError) as ei:
            bc.bc_probe_drift_noalloc(16, 16, n_max + 1, dt, 16, 0)
        assert ei.value.status == bc.ERR_INVALID_ARG
        assert str(n_max) in str(ei.value)
