"""The no-allocation probe drift (bc_probe_drift_noalloc).

Some callers cannot call cudaMalloc, nor let a library allocate for them: code inside a host
framework that owns all device memory, or a latency-bound loop that cannot take the implicit
device synchronisation of an allocation.  For them the library offers the probe drift with its
reduction scratch in the library's own static device memory.  These tests call it through the
C ABI and check it against the handle-based bc_probe_drift, on two calls in a row, with the
tolerance the drift tests use.  The file is named to be collected last.
"""
import numpy as np
import pytest
import torch

from paper_2608_28670_gb300 import barycache as bc
from paper_2608_28670_gb300 import synth

RTOL = 2e-6          # the tolerance of the drift parity tests


@pytest.fixture(scope="module")
def built():
    import __graft_entry__
    __graft_entry__.build_libraries()


def _inputs(n, dt, seed):
    rng = np.random.default_rng(seed)
    prev = rng.standard_normal(n).astype(np.float32)
    cur = prev + 0.05 * rng.standard_normal(n).astype(np.float32)
    if dt == bc.DTYPE_BF16:
        prev, cur = synth.f32_to_bf16_bits(prev), synth.f32_to_bf16_bits(cur)
        return (torch.from_numpy(cur.view(np.int16)).cuda(),
                torch.from_numpy(prev.view(np.int16)).cuda())
    return torch.from_numpy(cur).cuda(), torch.from_numpy(prev).cuda()


@pytest.mark.gpu
@pytest.mark.parametrize("dt", [bc.DTYPE_BF16, bc.DTYPE_F32])
@pytest.mark.parametrize("n", [0, 5, 8, 4099, 1_048_576 + 9, 40_000_000 + 3])
def test_no_alloc_drift_matches_handle_drift_twice(built, dt, n):
    torch.cuda.set_device(0)
    cur, prev = _inputs(n, dt, seed=n + 7 * dt)
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
        for k in range(2):
            np.testing.assert_allclose(o[k], r, rtol=RTOL, atol=0.0)
    finally:
        bc.bc_cache_destroy(h)


def test_no_alloc_drift_rejects_sizes_beyond_its_scratch(built):
    # The size check happens on the host before any device work, so no GPU is needed.
    for dt, n_max in [(bc.DTYPE_BF16, 1 << 29), (bc.DTYPE_F32, 1 << 28)]:
        with pytest.raises(bc.BaryCacheError) as ei:
            bc.bc_probe_drift_noalloc(16, 16, n_max + 1, dt, 16, 0)
        assert ei.value.status == bc.ERR_INVALID_ARG
        assert str(n_max) in str(ei.value)
