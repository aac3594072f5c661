"""Maximum sizes: one layer of more than 2^31 elements (its byte offsets pass 4 GiB).

Element, vector, tile and byte indices past 32 bits must all be carried in 64-bit
arithmetic.  A single bf16 layer of 2^31 + 3 * 8192 + 5 elements (4.3 GB per slot; about
22 GB on the device in all) goes through the zero-copy push, both forecast kernels, the
push copy and the probe drift.  Forecast outputs are checked against the fp64 oracle on
sampled elements around the 2^31 element (= 2^32 byte) boundary, the ragged tail and
random positions; the two kernels must agree on every element; the push copy must be
byte-exact everywhere; the drift is checked against the oracle summed over chunks, and
through a property that holds exactly at any size.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2608_28670_gb300 import barycache as bc
from paper_2608_28670_gb300 import synth
from tests.gpu_helpers import assert_close, device_view, oracle_weights, stream

pytestmark = pytest.mark.gpu

N = 2 ** 31 + 3 * 8192 + 5
TIMES = [0.7, 0.65, 0.6]            # pushed oldest first
T_NEW = 0.55
SEED = 77


@pytest.fixture(scope="module")
def big():
    import __graft_entry__
    __graft_entry__.build_libraries()
    torch.cuda.set_device(0)
    torch.cuda.empty_cache()
    free, _ = torch.cuda.mem_get_info()
    need = 6 * N * 2 + 2 * 10 ** 9
    if free < need:
        pytest.skip(f"needs {need / 1e9:.0f} GB free, have {free / 1e9:.0f} GB")
    h = bc.bc_cache_create([N], 3, bc.DTYPE_BF16)
    try:
        for i, t in enumerate(TIMES):
            slot = bc.bc_cache_next_slot_ptrs(h, 1)[0]
            synth.fill_device(slot, bc.DTYPE_BF16, N, seed=SEED, tensor_id=0, step_id=i,
                              tau=t, degree=2, noise_std=1e-2, hidden=3072,
                              stream=stream())
            torch.cuda.synchronize()
            bc.bc_cache_commit(h, t)
        yield h
    finally:
        bc.bc_cache_destroy(h)
        torch.cuda.empty_cache()


def sample_indices(rng) -> torch.Tensor:
    edge = 2 ** 31
    fixed = [0, 1, 8191, 8192, N // 2, N - 6, N - 5, N - 1]
    fixed += list(range(edge - 40, edge + 40))
    fixed += [edge - 8192 - 1, edge - 8192, edge + 8192, edge + 8193]
    idx = np.unique(np.concatenate([np.array(fixed, dtype=np.int64),
                                    rng.integers(0, N, 4096)]))
    return torch.from_numpy(idx).cuda()


def test_forecast_past_2_pow_31_elements_both_kernels(big):
    h = big
    out = torch.empty(N, dtype=torch.int16, device="cuda")
    idx = sample_indices(np.random.default_rng(5))
    assert bc.bc_cache_nodes(h) == [0.6, 0.65, 0.7]
    slots = [bc.bc_cache_slot_ptrs(h, j, 1)[0] for j in range(3)]   # newest first
    F = [device_view(p, N, bc.DTYPE_BF16)[idx].cpu().numpy().view(np.uint16) for p in slots]
    W = oracle_weights([0.6, 0.65, 0.7], T_NEW, bc.MODE_PAPER)
    ref, bound = oracle.combine(F, W)
    first = None
    for kern in (bc.KERNEL_REGISTER, bc.KERNEL_PIPELINE):
        bc.bc_cache_set_kernel(h, kern)
        out.fill_(0x5A5A)
        bc.bc_forecast(h, T_NEW, [out.data_ptr()], bc.DTYPE_BF16, stream())
        torch.cuda.synchronize()
        got = out[idx].cpu().numpy().view(np.uint16)
        assert_close(got, ref, bound, bc.DTYPE_BF16, f"kernel {kern}")
        if first is None:
            first = out.clone()
    assert torch.equal(first, out)               # every element, both kernels
    del first
    bc.bc_cache_set_kernel(h, bc.KERNEL_AUTO)
    bc.bc_cache_check(h)


def test_probe_drift_past_2_pow_31_elements(big):
    h = big
    assert bc.bc_cache_nodes(h) == [0.6, 0.65, 0.7]
    s0, s1 = [bc.bc_cache_slot_ptrs(h, j, 1)[0] for j in range(2)]   # nodes 0.6, 0.65
    out = torch.empty(3, dtype=torch.float64, device="cuda")
    bc.bc_probe_drift(h, s0, s1, N, bc.DTYPE_BF16, out.data_ptr(), stream())
    torch.cuda.synchronize()
    got = out.cpu().numpy()
    # The oracle over chunks of 2^28 elements, the chunk sums added in fp64.
    ref = np.zeros(2)
    step = 2 ** 28
    cur, prev = device_view(s0, N, bc.DTYPE_BF16), device_view(s1, N, bc.DTYPE_BF16)
    for a in range(0, N, step):
        b = min(N, a + step)
        c = cur[a:b].cpu().numpy().view(np.uint16)
        p = prev[a:b].cpu().numpy().view(np.uint16)
        ref += oracle.drift(c, p)[:2]
    np.testing.assert_allclose(got[:2], ref, rtol=2e-6, atol=0.0)
    np.testing.assert_allclose(got[2], ref[0] / ref[1], rtol=4e-6)

    # Exact at any size: with cur = -prev every |cur - prev| is exactly 2 |prev| (a power
    # of two scale), so the two sums see the same additions scaled by 2 and out[2] == 2.
    neg = torch.bitwise_xor(prev, torch.tensor(-32768, dtype=torch.int16, device="cuda"))
    bc.bc_probe_drift(h, neg.data_ptr(), s1, N, bc.DTYPE_BF16, out.data_ptr(), stream())
    torch.cuda.synchronize()
    o = out.cpu().numpy()
    assert o[0] == 2.0 * o[1] and o[2] == 2.0
    np.testing.assert_allclose(o[1], ref[1], rtol=2e-6)
    del neg
    # The no-allocation variant rejects this size before enqueueing anything.
    with pytest.raises(bc.BaryCacheError) as ei:
        bc.bc_probe_drift_noalloc(s0, s1, N, bc.DTYPE_BF16, out.data_ptr(), stream())
    assert ei.value.status == bc.ERR_INVALID_ARG


def test_push_copy_past_4_gib_is_byte_exact_both_kernels(big):
    h = big
    src = torch.empty(N, dtype=torch.int16, device="cuda")
    synth.fill_device(src.data_ptr(), bc.DTYPE_BF16, N, seed=SEED + 1, tensor_id=0,
                      step_id=9, tau=0.5, degree=2, noise_std=1e-2, hidden=3072,
                      stream=stream())
    src[N - 1] = -1                              # a NaN payload in the last element
    torch.cuda.synchronize()
    try:
        for kern, t in ((bc.KERNEL_REGISTER, 0.5), (bc.KERNEL_PIPELINE, 0.45)):
            bc.bc_cache_set_kernel(h, kern)
            bc.bc_cache_push(h, [src.data_ptr()], t, stream())
            torch.cuda.synchronize()
            bc.bc_cache_check(h)
            got = device_view(bc.bc_cache_slot_ptrs(h, 0, 1)[0], N, bc.DTYPE_BF16)
            assert torch.equal(got, src)
        assert bc.bc_cache_nodes(h) == [0.45, 0.5, 0.6]
        bc.bc_cache_set_kernel(h, bc.KERNEL_AUTO)
    finally:
        del src
        torch.cuda.empty_cache()
