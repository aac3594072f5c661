"""Failure behaviour of the C ABI on a GPU: every fault is injected on the host side (bad
arguments, wrong call order, a device allocation the GPU cannot satisfy) and must come back
as a status code with a message, leaving the context usable."""
import pytest
import torch

from paper_2608_28670_gb300 import barycache as bc
from tests.gpu_helpers import device_view

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def built():
    import __graft_entry__
    __graft_entry__.build_libraries()
    torch.cuda.set_device(0)


def _status(fn, *args):
    with pytest.raises(bc.BaryCacheError) as ei:
        fn(*args)
    assert bc.lib().bc_last_error().decode()
    return ei.value.status


def s():
    return torch.cuda.current_stream().cuda_stream


def test_forecast_before_any_push_is_not_ready():
    h = bc.bc_cache_create([1024], 3, bc.DTYPE_BF16)
    try:
        out = torch.empty(1024, dtype=torch.bfloat16, device="cuda")
        assert _status(bc.bc_forecast, h, 0.5, [out.data_ptr()], bc.DTYPE_BF16, s()) == \
            bc.ERR_NOT_READY
        assert _status(bc.bc_coefficients, h, 0.5) == bc.ERR_NOT_READY
        assert _status(bc.bc_forecast_flat, h, 0.5, out.data_ptr(), s()) == bc.ERR_NOT_READY
    finally:
        bc.bc_cache_destroy(h)


def test_duplicate_nodes_and_ring_eviction():
    h = bc.bc_cache_create([256], 2, bc.DTYPE_F32)
    try:
        x = torch.zeros(256, device="cuda")
        bc.bc_cache_push(h, [x.data_ptr()], 0.9, s())
        assert _status(bc.bc_cache_push, h, [x.data_ptr()], 0.9, s()) == bc.ERR_DUPLICATE_NODE
        bc.bc_cache_push(h, [x.data_ptr()], 0.8, s())
        # window full (0.8, 0.9): pushing 0.9 again evicts 0.9 first, so it is not a duplicate
        bc.bc_cache_push(h, [x.data_ptr()], 0.9, s())
        assert bc.bc_cache_nodes(h) == [0.9, 0.8]
        # 0.8 is the oldest and would be evicted by this commit: allowed; 0.9 stays: duplicate
        assert _status(bc.bc_cache_commit, h, 0.9) == bc.ERR_DUPLICATE_NODE
        assert _status(bc.bc_cache_commit, h, float("nan")) == bc.ERR_INVALID_ARG
        bc.bc_cache_reset(h)
        assert bc.bc_cache_nodes(h) == []
        assert bc.bc_cache_stats(h)["pushes"] == 3
    finally:
        bc.bc_cache_destroy(h)


def test_pointer_checks():
    h = bc.bc_cache_create([4096, 100], 2, bc.DTYPE_BF16)
    try:
        x = torch.zeros(8192, dtype=torch.bfloat16, device="cuda")
        p = x.data_ptr()
        assert _status(bc.bc_cache_push, h, [p + 2, p], 0.5, s()) == bc.ERR_ALIGNMENT
        assert _status(bc.bc_cache_push, h, [p, 0], 0.5, s()) == bc.ERR_INVALID_ARG
        slot = bc.bc_cache_next_slot_ptrs(h, 2)
        assert _status(bc.bc_cache_push, h, [slot[0], p], 0.5, s()) == bc.ERR_INVALID_ARG
        bc.bc_cache_push(h, [p, p], 0.5, s())
        assert _status(bc.bc_forecast, h, 0.4, [p + 16 + 2, None], bc.DTYPE_BF16, s()) == \
            bc.ERR_ALIGNMENT
        live = bc.bc_cache_slot_ptrs(h, 0, 2)
        assert _status(bc.bc_forecast, h, 0.4, [live[0], None], bc.DTYPE_BF16, s()) == \
            bc.ERR_INVALID_ARG                                   # output inside the arena
        assert _status(bc.bc_forecast, h, 0.4, [p, None], 7, s()) == bc.ERR_INVALID_ARG
        assert _status(bc.bc_forecast_step, h, 0.4, -0.1, [p, None], bc.DTYPE_BF16, 0, p,
                       bc.DTYPE_F32, s()) == bc.ERR_INVALID_ARG       # output aliases x
        assert _status(bc.bc_forecast_step, h, 0.4, -0.1, [None, None], bc.DTYPE_BF16, 5, p,
                       bc.DTYPE_F32, s()) == bc.ERR_INVALID_ARG       # no such layer
        assert _status(bc.bc_forecast, h, float("inf"), [p, None], bc.DTYPE_BF16, s()) == \
            bc.ERR_INVALID_ARG
        assert _status(bc.bc_cache_slot_ptrs, h, 1, 2) == bc.ERR_INVALID_ARG
        # the flat push: one slot image of 8192 + 256 bytes
        assert bc.bc_cache_layout(h)[-1] <= x.numel() * 2
        assert _status(bc.bc_cache_push_flat, h, p + 2, 0.3, s()) == bc.ERR_ALIGNMENT
        assert _status(bc.bc_cache_push_flat, h, 0, 0.3, s()) == bc.ERR_INVALID_ARG
        nxt = bc.bc_cache_next_slot_ptrs(h, 2)
        assert _status(bc.bc_cache_push_flat, h, nxt[0], 0.3, s()) == bc.ERR_INVALID_ARG
        assert _status(bc.bc_cache_push_flat, h, p, 0.5, s()) == bc.ERR_DUPLICATE_NODE
        assert _status(bc.bc_cache_push_flat, h, p, float("nan"), s()) == bc.ERR_INVALID_ARG
        assert bc.bc_cache_nodes(h) == [0.5]                     # nothing was pushed
        bc.bc_cache_push_flat(h, p, 0.3, s())
        assert bc.bc_cache_nodes(h) == [0.3, 0.5]
    finally:
        bc.bc_cache_destroy(h)
    torch.cuda.synchronize()                     # the context is still usable


def test_destroyed_handle_is_rejected():
    h = bc.bc_cache_create([64], 2, bc.DTYPE_F32)
    bc.bc_cache_destroy(h)
    assert _status(bc.bc_cache_bytes, h) == bc.ERR_BAD_HANDLE
    assert _status(bc.bc_cache_destroy, h) == bc.ERR_BAD_HANDLE
    assert _status(bc.bc_forecast, h, 0.1, [None], bc.DTYPE_F32, s()) == bc.ERR_BAD_HANDLE


def test_device_out_of_memory_is_a_status():
    free, total = torch.cuda.mem_get_info()
    numel = (total // 2) * 2                     # K = 2 slots of `total` bytes of bf16 each
    assert _status(bc.bc_cache_create, [numel // 2], 2, bc.DTYPE_BF16) in (bc.ERR_OOM,)
    h = bc.bc_cache_create([1024], 2, bc.DTYPE_BF16)   # the device still allocates afterwards
    bc.bc_cache_destroy(h)


def test_degenerate_weights_status():
    h = bc.bc_cache_create([64], 2, bc.DTYPE_F32,
                           bc.make_params(mode=bc.MODE_PAPER, delta=1.0, eta=0.0))
    try:
        x = torch.zeros(64, device="cuda")
        bc.bc_cache_push(h, [x.data_ptr()], 0.02, s())
        bc.bc_cache_push(h, [x.data_ptr()], 0.01, s())
        out = torch.empty(64, device="cuda")
        assert _status(bc.bc_forecast, h, 0.0, [out.data_ptr()], bc.DTYPE_F32, s()) == \
            bc.ERR_DEGENERATE_WEIGHTS
    finally:
        bc.bc_cache_destroy(h)


@pytest.mark.parametrize("K", [3, 4])
@pytest.mark.parametrize("flat", [False, True])
def test_pipeline_wait_timeout_is_reported_and_recovers(flat, K):
    """Failure detection on the device: the test hook leaves each CTA's first pipeline stage
    unarmed, so the forecast kernel's bounded wait runs out (about a second); the launch
    returns, bc_cache_check reports BC_ERR_DEVICE_TIMEOUT once, and the next forecast on the
    same handle and context is correct.  The drain after the timeout skips the unarmed stage,
    so the whole launch gives up after one wait limit, not two."""
    import time
    import numpy as np
    import oracle
    from paper_2608_28670_gb300 import synth
    from tests.gpu_helpers import assert_close, to_device, to_host
    numels = [100_000, 3 * 8192 + 5]
    times = [0.9, 0.85, 0.8, 0.775][:K]
    feats = synth.host_trajectories([(n,) for n in numels], times, dtype="bf16", seed=44)
    h = bc.bc_cache_create(numels, K, bc.DTYPE_BF16)
    try:
        for t, per in zip(times, feats):
            dev = [to_device(f) for f in per]
            bc.bc_cache_push(h, [d.data_ptr() for d in dev], t, s())
            torch.cuda.synchronize()
        bc.bc_cache_check(h)
        offs = bc.bc_cache_layout(h, 2)
        flat_out = torch.empty(offs[-1] // 2, dtype=torch.int16, device="cuda")
        outs = [torch.empty(n, dtype=torch.int16, device="cuda") for n in numels]

        def forecast():
            if flat:
                bc.bc_forecast_flat(h, 0.75, flat_out.data_ptr(), s())
            else:
                bc.bc_forecast(h, 0.75, [o.data_ptr() for o in outs], bc.DTYPE_BF16, s())

        bc.bc_cache_inject_fault(h, 1)
        t0 = time.perf_counter()
        forecast()
        assert _status(bc.bc_cache_check, h) == bc.ERR_DEVICE_TIMEOUT
        assert 0.5 < time.perf_counter() - t0 < 1.9
        bc.bc_cache_check(h)                         # reported once, then clear
        forecast()                                   # the handle and context still work
        bc.bc_cache_check(h)
        torch.cuda.synchronize()
        W = oracle.paper_weights(times[::-1], 0.75)
        nf = feats[::-1]
        host_flat = to_host(flat_out, bc.DTYPE_BF16)
        for l, n in enumerate(numels):
            got = host_flat[offs[l] // 2: offs[l] // 2 + n] if flat else to_host(outs[l], bc.DTYPE_BF16)
            ref, bound = oracle.combine([f[l] for f in nf], W)
            assert_close(got, ref, bound, bc.DTYPE_BF16, f"after recovery, layer {l}")
    finally:
        bc.bc_cache_destroy(h)


def test_drift_pipeline_wait_timeout_is_reported_and_recovers():
    """The same failure detection for the probe drift's pipeline form: with its first stage
    left unarmed every CTA gives up, out[] reads NaN, bc_cache_check reports the timeout once,
    and the next drift on the handle is right."""
    import time
    import numpy as np
    import oracle
    from tests.gpu_helpers import to_device
    n = 8192 * 300 + 5
    rng = np.random.default_rng(3)
    prev = rng.standard_normal(n).astype(np.float32)
    cur = prev + 0.1 * rng.standard_normal(n).astype(np.float32)
    c, p = to_device(cur), to_device(prev)
    h = bc.bc_cache_create([16], 2, bc.DTYPE_F32)
    bc.bc_cache_set_kernel(h, bc.KERNEL_PIPELINE)
    try:
        out = torch.zeros(3, dtype=torch.float64, device="cuda")
        bc.bc_cache_inject_fault(h, 2)
        t0 = time.perf_counter()
        bc.bc_probe_drift(h, c.data_ptr(), p.data_ptr(), n, bc.DTYPE_F32, out.data_ptr(), s())
        assert _status(bc.bc_cache_check, h) == bc.ERR_DEVICE_TIMEOUT
        assert 0.5 < time.perf_counter() - t0 < 1.9
        assert np.isnan(out.cpu().numpy()).all()
        bc.bc_cache_check(h)
        bc.bc_probe_drift(h, c.data_ptr(), p.data_ptr(), n, bc.DTYPE_F32, out.data_ptr(), s())
        bc.bc_cache_check(h)
        np.testing.assert_allclose(out.cpu().numpy(), oracle.drift(cur, prev), rtol=2e-6)
        assert bc.bc_cache_stats(h)["pipeline_launches"] == 2
    finally:
        bc.bc_cache_destroy(h)


@pytest.mark.parametrize("flat", [False, True], ids=["per_layer", "flat"])
def test_push_pipeline_wait_timeout_is_reported_and_recovers(flat):
    """The push copy's pipeline form under the same test hook: the launch gives up, the
    check reports it once, and the next push on the handle copies every byte."""
    import time
    n = 16384 * 40 + 7
    src = torch.arange(n + 57, dtype=torch.float32, device="cuda")   # a whole 256-byte slot

    def push(t):
        if flat:
            bc.bc_cache_push_flat(h, src.data_ptr(), t, s())
        else:
            bc.bc_cache_push(h, [src.data_ptr()], t, s())

    h = bc.bc_cache_create([n], 2, bc.DTYPE_F32)
    bc.bc_cache_set_kernel(h, bc.KERNEL_PIPELINE)
    try:
        assert bc.bc_cache_layout(h)[-1] == src.numel() * 4
        bc.bc_cache_inject_fault(h, 3)
        t0 = time.perf_counter()
        push(0.9)
        assert _status(bc.bc_cache_check, h) == bc.ERR_DEVICE_TIMEOUT
        assert 0.5 < time.perf_counter() - t0 < 1.9
        bc.bc_cache_check(h)
        bc.bc_cache_reset(h)
        push(0.9)
        bc.bc_cache_check(h)
        got = device_view(bc.bc_cache_slot_ptrs(h, 0, 1)[0], n, bc.DTYPE_F32)
        assert torch.equal(got, src[:n])
        assert bc.bc_cache_stats(h)["pipeline_launches"] == 2
    finally:
        bc.bc_cache_destroy(h)


def test_check_is_clean_after_normal_launches_and_rejects_unknown_choices():
    h = bc.bc_cache_create([4096], 2, bc.DTYPE_BF16)
    try:
        assert _status(bc.bc_cache_inject_fault, h, 4) == bc.ERR_INVALID_ARG
        assert _status(bc.bc_cache_inject_fault, h, -1) == bc.ERR_INVALID_ARG
        assert _status(bc.bc_cache_set_kernel, h, 3) == bc.ERR_INVALID_ARG
        bc.bc_cache_check(h)
    finally:
        bc.bc_cache_destroy(h)


def test_binding_rejects_per_layer_lists_of_the_wrong_length():
    # The C calls read exactly n_layers pointers; the binding must stop shorter lists.
    h = bc.bc_cache_create([256, 512], 2, bc.DTYPE_F32)
    try:
        assert bc.bc_cache_info(h) == (2, 2, bc.DTYPE_F32)
        x = torch.zeros(512, device="cuda")
        assert _status_py(bc.bc_cache_push, h, [x.data_ptr()], 0.5, s()) == bc.ERR_INVALID_ARG
        bc.bc_cache_push(h, [x.data_ptr(), x.data_ptr()], 0.5, s())
        assert _status_py(bc.bc_forecast, h, 0.4, [x.data_ptr()], bc.DTYPE_F32, s()) == \
            bc.ERR_INVALID_ARG
        assert _status_py(bc.bc_forecast, h, 0.4, [None] * 3, bc.DTYPE_F32, s()) == \
            bc.ERR_INVALID_ARG
        assert len(bc.bc_cache_next_slot_ptrs(h)) == 2 and len(bc.bc_cache_layout(h)) == 3
    finally:
        bc.bc_cache_destroy(h)


def _status_py(fn, *args):
    with pytest.raises(bc.BaryCacheError) as ei:
        fn(*args)
    return ei.value.status
