"""GPU parity of the grouped forecast, the push copy and the fused Euler step.

Every case builds seeded host features (numpy), pushes them through the C ABI, runs the
CUDA path and compares each output element with the fp64 oracle on the same stored inputs:
|gpu - oracle| <= 1e-5 * sum_j |W_j||F_j| for fp32 output, 2^-8 * sum_j |W_j||F_j| for bf16
(and |x| + |dt| sum_j |W_j||V_j| for the Euler state).  Sizes span several tiles and
ragged tails while keeping the oracle fast.
"""
from math import prod

import numpy as np
import pytest
import torch

import oracle
from paper_2608_28670_gb300 import barycache as bc
from paper_2608_28670_gb300 import synth
from tests.gpu_helpers import (as_f64, assert_close, device_view, empty_out, oracle_weights,
                               stream, to_device, to_host)

pytestmark = pytest.mark.gpu

DT_NAME = {bc.DTYPE_F32: "f32", bc.DTYPE_BF16: "bf16"}
# A tile holds 16 KiB of each history slot (32 KiB at K = 4 in the register kernel, 8 KiB in
# small launches): 8192 bf16 / 4096 f32 elements.
RAGGED = [1, 7, 8, 9, 4095, 4096, 4097, 8191, 8192, 8193, 3 * 8192 + 5, 100_003]


@pytest.fixture(scope="module", autouse=True)
def built():
    import __graft_entry__
    __graft_entry__.build_libraries()
    torch.cuda.set_device(0)


KERNELS = [bc.KERNEL_REGISTER, bc.KERNEL_PIPELINE]
KNAME = {bc.KERNEL_REGISTER: "register", bc.KERNEL_PIPELINE: "pipeline"}


def run_case(numels, K, n_push, in_dt, out_dt, params, t_new, push_times, seed,
             zero_copy=False, pad=64, kernel=bc.KERNEL_AUTO):
    shapes = [(n,) for n in numels]
    taus = list(push_times)
    feats = synth.host_trajectories(shapes, taus, dtype=DT_NAME[in_dt], degree=2,
                                    noise_std=1e-2, seed=seed)
    h = bc.bc_cache_create(numels, K, in_dt, params)
    bc.bc_cache_set_kernel(h, kernel)
    try:
        for i in range(n_push):
            if zero_copy:
                slots = bc.bc_cache_next_slot_ptrs(h, len(numels))
                for l, n in enumerate(numels):
                    if n:
                        device_view(slots[l], n, in_dt).copy_(to_device(feats[i][l]))
                bc.bc_cache_commit(h, push_times[i])
            else:
                dev = [to_device(f) for f in feats[i]]
                bc.bc_cache_push(h, [d.data_ptr() for d in dev], push_times[i], stream())
                torch.cuda.synchronize()   # `dev` may be freed after this
        outs = [empty_out(n, out_dt, pad) for n in numels]
        for o in outs:
            o.fill_(0x5A5A if out_dt == bc.DTYPE_BF16 else 7.25)
        ptrs = [o.data_ptr() + pad * o.element_size() for o in outs]
        bc.bc_forecast(h, t_new, ptrs, out_dt, stream())
        torch.cuda.synchronize()
        m = min(n_push, K)
        nodes = list(reversed(push_times[:n_push]))[:m]
        got_nodes = bc.bc_cache_nodes(h)
        assert got_nodes == nodes
        W = oracle_weights(nodes, t_new, params.mode, lam=params.lambda_,
                           delta=params.delta if params.delta > 0 else None,
                           C=params.clip_C, eta=params.eta)
        newest_first = [feats[i] for i in range(n_push - 1, n_push - 1 - m, -1)]
        for l, n in enumerate(numels):
            host = to_host(outs[l], out_dt)
            canary = 0x5A5A if out_dt == bc.DTYPE_BF16 else np.float32(7.25)
            assert np.all(host[:pad] == canary) and np.all(host[pad + n:] == canary), \
                f"layer {l}: write outside the output"
            if n == 0:
                continue
            ref, bound = oracle.combine([f[l] for f in newest_first], W)
            assert_close(host[pad:pad + n], ref, bound, out_dt, f"layer {l} numel {n}")
        bc.bc_cache_check(h)
        return h
    except Exception:
        bc.bc_cache_destroy(h)
        raise


@pytest.mark.parametrize("kernel", KERNELS, ids=KNAME.get)
@pytest.mark.parametrize("in_dt", [bc.DTYPE_BF16, bc.DTYPE_F32])
@pytest.mark.parametrize("out_dt", [bc.DTYPE_BF16, bc.DTYPE_F32])
@pytest.mark.parametrize("K", [1, 2, 3, 4])
def test_ragged_layers_all_dtypes(in_dt, out_dt, K, kernel):
    times = [0.9 - 0.05 * i for i in range(K)]
    h = run_case(RAGGED, K, K, in_dt, out_dt, bc.make_params(), times[-1] - 0.05, times,
                 seed=K * 10 + in_dt * 2 + out_dt, kernel=kernel)
    bc.bc_cache_destroy(h)


@pytest.mark.parametrize("kernel", KERNELS, ids=KNAME.get)
@pytest.mark.parametrize("K", [2, 3, 4])
@pytest.mark.parametrize("mode", [bc.MODE_EXACT, bc.MODE_PAPER])
def test_partial_and_rotating_window(K, mode, kernel):
    # Fewer pushes than K (m < K), exactly K, and K + 3 (the ring has wrapped).
    for n_push in (1, K - 1, K, K + 3):
        if n_push < 1:
            continue
        times = [980.0 - 20.0 * i for i in range(n_push)]
        h = run_case([5000, 70_001], K, n_push, bc.DTYPE_BF16, bc.DTYPE_BF16,
                     bc.make_params(mode=mode), times[-1] - 20.0, times, seed=n_push,
                     kernel=kernel)
        bc.bc_cache_destroy(h)


@pytest.mark.parametrize("kernel", KERNELS, ids=KNAME.get)
@pytest.mark.parametrize("lam,delta,C", [(0.0, 0.0, 10.0), (0.5, 0.0, 10.0), (1.0, 0.0, 10.0),
                                         (0.0, 0.7, 2.0), (0.2, 1.0, 10.0)])
def test_weight_parameters_flow_time(lam, delta, C, kernel):
    # Flow-matching time in [0, 1]: the clip of Eq. 10 is active at this spacing.
    times = [1.0, 25 / 28, 22 / 28]
    h = run_case([33_333, 8192], 3, 3, bc.DTYPE_BF16, bc.DTYPE_F32,
                 bc.make_params(lam=lam, delta=delta, clip_C=C), 21 / 28, times, seed=5,
                 kernel=kernel)
    bc.bc_cache_destroy(h)


@pytest.mark.parametrize("kernel", KERNELS, ids=KNAME.get)
def test_zero_copy_push(kernel):
    times = [0.8, 0.7, 0.6, 0.5, 0.4]
    h = run_case([12_345, 1, 65_536], 3, 5, bc.DTYPE_BF16, bc.DTYPE_BF16, bc.make_params(),
                 0.35, times, seed=11, zero_copy=True, kernel=kernel)
    bc.bc_cache_destroy(h)


@pytest.mark.parametrize("K", [1, 2, 3, 4])
@pytest.mark.parametrize("in_dt", [bc.DTYPE_BF16, bc.DTYPE_F32])
@pytest.mark.parametrize("out_dt", [bc.DTYPE_BF16, bc.DTYPE_F32])
def test_register_and_pipeline_kernels_agree_bitwise(K, in_dt, out_dt):
    # The two kernels apply the same fp32 FMA chain; only where the history bytes travel
    # through differs, so every output and the updated latent must match bit for bit.
    numels = RAGGED + [3 * 8192 * 8 + 17]
    times = [0.9 - 0.05 * i for i in range(K)]
    feats = synth.host_trajectories([(n,) for n in numels], times, dtype=DT_NAME[in_dt], seed=K)
    h = bc.bc_cache_create(numels, K, in_dt)
    try:
        for t, per in zip(times, feats):
            dev = [to_device(f) for f in per]
            bc.bc_cache_push(h, [d.data_ptr() for d in dev], t, stream())
            torch.cuda.synchronize()
        x0 = torch.linspace(-3, 3, numels[-1], device="cuda")
        results = []
        for kern in KERNELS:
            bc.bc_cache_set_kernel(h, kern)
            outs = [empty_out(n, out_dt) for n in numels[:-1]]
            x = x0.clone()
            bc.bc_forecast_update(h, times[-1] - 0.05, 0.99, -0.05, 0.0,
                                  [o.data_ptr() for o in outs] + [None], out_dt,
                                  len(numels) - 1, x.data_ptr(), bc.DTYPE_F32, None, stream())
            torch.cuda.synchronize()
            results.append([o.cpu() for o in outs] + [x.cpu()])
        bc.bc_cache_check(h)
        for a, b in zip(*results):
            assert torch.equal(a, b)
    finally:
        bc.bc_cache_destroy(h)


def test_exact_mode_node_hit_returns_the_node():
    times = [0.8, 0.7, 0.6]
    h = run_case([10_000], 3, 3, bc.DTYPE_F32, bc.DTYPE_F32, bc.make_params(mode=bc.MODE_EXACT),
                 0.7, times, seed=3)
    try:
        out = torch.empty(10_000, dtype=torch.float32, device="cuda")
        bc.bc_forecast(h, 0.7, [out.data_ptr()], bc.DTYPE_F32, stream())
        slot = device_view(bc.bc_cache_slot_ptrs(h, 1, 1)[0], 10_000, bc.DTYPE_F32)
        torch.cuda.synchronize()
        assert torch.equal(out, slot)
    finally:
        bc.bc_cache_destroy(h)


@pytest.mark.parametrize("kernel", KERNELS, ids=KNAME.get)
@pytest.mark.parametrize("dt", [bc.DTYPE_BF16, bc.DTYPE_F32])
def test_push_copy_is_byte_exact(kernel, dt):
    # Includes NaN payloads and -0.0: the push must move bytes, not values.  Layer sizes
    # span whole and ragged 32 KiB pipeline tiles, ends shorter than 16 bytes and a layer
    # smaller than one 16-byte group.
    eb = 2 if dt == bc.DTYPE_BF16 else 4
    numels = [3 * 8192 + 3, 3 * 8192 + 4, 16384 // eb * 5, 3, 100_003]
    rng = np.random.default_rng(1)
    src = []
    for n in numels:
        if dt == bc.DTYPE_BF16:
            bits = rng.integers(0, 2 ** 16, n, dtype=np.uint16)
            bits[:min(n, 4)] = [0x7FC1, 0xFFFF, 0x8000, 0x7F80][:min(n, 4)]
            src.append(to_device(bits))
        else:
            bits = rng.integers(0, 2 ** 32, n, dtype=np.uint64).astype(np.uint32)
            bits[:min(n, 3)] = [0x7FC00001, 0xFFFFFFFF, 0x80000000][:min(n, 3)]
            src.append(to_device(bits.view(np.float32)))
    h = bc.bc_cache_create(numels, 2, dt)
    bc.bc_cache_set_kernel(h, kernel)
    try:
        p0 = bc.bc_cache_stats(h)["pipeline_launches"]
        bc.bc_cache_push(h, [s.data_ptr() for s in src], 0.5, stream())
        torch.cuda.synchronize()
        bc.bc_cache_check(h)
        assert bc.bc_cache_stats(h)["pipeline_launches"] - p0 == \
            (1 if kernel == bc.KERNEL_PIPELINE else 0)
        slots = bc.bc_cache_slot_ptrs(h, 0, len(numels))
        for l, s in enumerate(src):
            got = device_view(slots[l], s.numel(), dt)
            if dt == bc.DTYPE_F32:
                assert torch.equal(got.view(torch.int32), s.view(torch.int32))
            else:
                assert torch.equal(got, s)
    finally:
        bc.bc_cache_destroy(h)


@pytest.mark.parametrize("kernel", KERNELS, ids=KNAME.get)
@pytest.mark.parametrize("dt", [bc.DTYPE_BF16, bc.DTYPE_F32])
def test_flat_push_copies_the_slot_image_byte_exact(kernel, dt):
    # bc_cache_push_flat copies a slot-shaped buffer (bc_cache_layout offsets, padding
    # included) in one launch: every byte of the slot equals the source, NaN payloads and
    # -0.0 included, and the forecasts then match those of per-layer pushes bit for bit.
    eb = 2 if dt == bc.DTYPE_BF16 else 4
    numels = [3 * 8192 + 3, 0, 16384 // eb * 5, 3, 100_003, 1]
    h = bc.bc_cache_create(numels, 3, dt)
    ref = bc.bc_cache_create(numels, 3, dt)
    bc.bc_cache_set_kernel(h, kernel)
    bc.bc_cache_set_kernel(ref, kernel)
    try:
        offs = bc.bc_cache_layout(h)
        rng = np.random.default_rng(41)
        images = []
        for k in range(3):
            if dt == bc.DTYPE_BF16:         # any bit pattern, specials planted up front
                bits = rng.integers(0, 2 ** 16, offs[-1] // 2, dtype=np.uint16)
                bits[:4] = [0x7FC1, 0xFFFF, 0x8000, 0x7F80]
                images.append(to_device(bits))
            else:                           # finite values except the planted specials
                v = rng.standard_normal(offs[-1] // 4).astype(np.float32)
                v.view(np.uint32)[:3] = [0x7FC00001, 0xFFFFFFFF, 0x80000000]
                images.append(to_device(v))
        times = [0.9, 0.85, 0.8]
        p0 = bc.bc_cache_stats(h)
        for k, t in enumerate(times):
            bc.bc_cache_push_flat(h, images[k].data_ptr(), t, stream())
            bc.bc_cache_push(ref, [images[k].data_ptr() + offs[l] if n else 0
                                   for l, n in enumerate(numels)], t, stream())
        torch.cuda.synchronize()
        bc.bc_cache_check(h)
        p1 = bc.bc_cache_stats(h)
        assert p1["kernel_launches"] - p0["kernel_launches"] == 3
        assert p1["pipeline_launches"] - p0["pipeline_launches"] == \
            (3 if kernel == bc.KERNEL_PIPELINE else 0)
        assert p1["table_uploads"] == p0["table_uploads"]
        assert bc.bc_cache_nodes(h) == [0.8, 0.85, 0.9]
        for j in range(3):
            base = bc.bc_cache_slot_ptrs(h, j)[0]
            whole = device_view(base, offs[-1] // eb, dt)
            want = images[2 - j]
            if dt == bc.DTYPE_F32:
                assert torch.equal(whole.view(torch.int32), want.view(torch.int32))
            else:
                assert torch.equal(whole, want)
        outs = {c: [empty_out(n, dt) for n in numels] for c in (h, ref)}
        for c in (h, ref):
            bc.bc_forecast(c, 0.75, [o.data_ptr() if n else None
                                     for o, n in zip(outs[c], numels)], dt, stream())
        torch.cuda.synchronize()
        for a, b, n in zip(outs[h], outs[ref], numels):
            if dt == bc.DTYPE_F32:
                assert torch.equal(a[:n].view(torch.int32), b[:n].view(torch.int32))
            else:
                assert torch.equal(a[:n], b[:n])
    finally:
        bc.bc_cache_destroy(h)
        bc.bc_cache_destroy(ref)


def test_null_outputs_skip_layers_and_window_forecast():
    numels = [8192 * 3, 1000, 77_777, 64]
    times = [0.9, 0.8, 0.7]
    h = run_case(numels, 3, 3, bc.DTYPE_BF16, bc.DTYPE_BF16, bc.make_params(), 0.65, times, seed=8)
    try:
        outs = [empty_out(n, bc.DTYPE_BF16) for n in numels]
        for o in outs:
            o.fill_(123)
        ptrs = [outs[0].data_ptr(), None, outs[2].data_ptr(), None]
        before = bc.bc_cache_stats(h)["kernel_launches"]
        bc.bc_forecast(h, 0.65, ptrs, bc.DTYPE_BF16, stream())
        torch.cuda.synchronize()
        assert bc.bc_cache_stats(h)["kernel_launches"] == before + 1
        assert torch.all(outs[1] == 123) and torch.all(outs[3] == 123)
        assert not torch.all(outs[0] == 123)
        # no output at all: nothing is launched
        bc.bc_forecast(h, 0.65, [None] * 4, bc.DTYPE_BF16, stream())
        assert bc.bc_cache_stats(h)["kernel_launches"] == before + 1
    finally:
        bc.bc_cache_destroy(h)


def test_many_layers_one_launch_through_the_device_table():
    # 1100 tiny ragged layers: more than one parameter block holds, so the layer table goes to
    # the handle's device copy and the forecast is one launch (run_case checks every layer
    # against the oracle).  The table is uploaded once for a set of outputs and again only
    # when the outputs change.
    numels = [(i * 37) % 301 + 1 for i in range(1100)]
    times = [0.9, 0.85]
    h = run_case(numels, 2, 2, bc.DTYPE_F32, bc.DTYPE_BF16, bc.make_params(), 0.8, times, seed=9)
    try:
        st0 = bc.bc_cache_stats(h)
        outs = [empty_out(n, bc.DTYPE_BF16) for n in numels]
        ptrs = [o.data_ptr() for o in outs]
        for _ in range(3):
            bc.bc_forecast(h, 0.8, ptrs, bc.DTYPE_BF16, stream())
        torch.cuda.synchronize()
        st1 = bc.bc_cache_stats(h)
        assert st1["kernel_launches"] - st0["kernel_launches"] == 3     # one per call
        assert st1["table_uploads"] - st0["table_uploads"] == 1          # new outputs: once
        first = [o.clone() for o in outs]
        ptrs2 = list(ptrs)
        ptrs2[5] = None                                                  # a different table
        outs[7].fill_(0)
        bc.bc_forecast(h, 0.8, ptrs2, bc.DTYPE_BF16, stream())
        bc.bc_forecast(h, 0.8, ptrs, bc.DTYPE_BF16, stream())
        torch.cuda.synchronize()
        assert bc.bc_cache_stats(h)["table_uploads"] - st0["table_uploads"] == 3
        for a, b in zip(first, outs):
            assert torch.equal(a, b)
        bc.bc_cache_check(h)
    finally:
        bc.bc_cache_destroy(h)


@pytest.mark.parametrize("kernel", KERNELS, ids=KNAME.get)
@pytest.mark.parametrize("dt", [bc.DTYPE_BF16, bc.DTYPE_F32])
def test_many_layer_push_is_one_byte_exact_launch(kernel, dt):
    # 1300 ragged layers (some empty, some shorter than a 16-byte group): the push copy reads
    # its table from the handle's device copy, one launch per push, uploaded again only when
    # the sources change; every byte lands (NaN payloads, -0.0 included).
    numels = [((i * 53) % 1201) * (i % 7 != 3) + (i % 5 == 0) for i in range(1300)]
    eb = 2 if dt == bc.DTYPE_BF16 else 4
    rng = np.random.default_rng(17)
    total = sum(numels)
    if dt == bc.DTYPE_BF16:
        bits = rng.integers(0, 2 ** 16, total, dtype=np.uint16)
    else:
        bits = rng.integers(0, 2 ** 32, total, dtype=np.uint64).astype(np.uint32)
    offs = np.cumsum([0] + numels)
    h = bc.bc_cache_create(numels, 2, dt)
    bc.bc_cache_set_kernel(h, kernel)
    try:
        srcs = []
        for l, n in enumerate(numels):
            seg = bits[offs[l]:offs[l + 1]]
            srcs.append(to_device(seg if dt == bc.DTYPE_BF16 else seg.view(np.float32))
                        if n else None)
        ptrs = [s_.data_ptr() if s_ is not None else 0 for s_ in srcs]
        st0 = bc.bc_cache_stats(h)
        bc.bc_cache_push(h, ptrs, 0.9, stream())
        bc.bc_cache_push(h, ptrs, 0.8, stream())          # same sources: no new upload
        torch.cuda.synchronize()
        bc.bc_cache_check(h)
        st1 = bc.bc_cache_stats(h)
        assert st1["kernel_launches"] - st0["kernel_launches"] == 2
        assert st1["table_uploads"] - st0["table_uploads"] == 1
        assert st1["pipeline_launches"] - st0["pipeline_launches"] == \
            (2 if kernel == bc.KERNEL_PIPELINE else 0)
        for j in (0, 1):
            slots = bc.bc_cache_slot_ptrs(h, j, len(numels))
            for l, n in enumerate(numels):
                if n:
                    got = device_view(slots[l], n, dt)
                    if dt == bc.DTYPE_F32:
                        assert torch.equal(got.view(torch.int32), srcs[l].view(torch.int32)), l
                    else:
                        assert torch.equal(got, srcs[l]), l
    finally:
        bc.bc_cache_destroy(h)


@pytest.mark.parametrize("kernel", KERNELS, ids=KNAME.get)
def test_many_layers_in_a_graph_carry_their_own_tables(kernel):
    # While the stream is captured, a forecast over more layers than one parameter block holds
    # is split into parameter-block launches, so the graph does not depend on the device table
    # that later calls rewrite.  Replaying it after an eager call with other outputs must
    # still write the captured outputs, bit for bit as the eager one-launch forecast.
    numels = [(i * 53) % 977 + 8 for i in range(2100)]
    times = [0.9, 0.85, 0.8]
    h = run_case(numels, 3, 3, bc.DTYPE_BF16, bc.DTYPE_BF16, bc.make_params(), 0.75, times,
                 seed=12, kernel=kernel)
    try:
        outs = [empty_out(n, bc.DTYPE_BF16) for n in numels]
        eager = [empty_out(n, bc.DTYPE_BF16) for n in numels]
        # first uses of the parameter-block launchers (1016- and 64-entry tables) outside the
        # capture, as the header asks
        for sel in (1000, 60):
            bc.bc_forecast(h, 0.75, [o.data_ptr() if l < sel else None
                                     for l, o in enumerate(eager)], bc.DTYPE_BF16, stream())
        bc.bc_forecast(h, 0.75, [o.data_ptr() for o in eager], bc.DTYPE_BF16, stream())
        torch.cuda.synchronize()
        g = torch.cuda.CUDAGraph()
        s = torch.cuda.Stream()
        with torch.cuda.stream(s):
            l0 = bc.bc_cache_stats(h)["kernel_launches"]
            with torch.cuda.graph(g, stream=s, capture_error_mode="thread_local"):
                bc.bc_forecast(h, 0.75, [o.data_ptr() for o in outs], bc.DTYPE_BF16,
                               s.cuda_stream)
            assert bc.bc_cache_stats(h)["kernel_launches"] - l0 == 3    # 1016 + 1016 + 68
        other = [empty_out(n, bc.DTYPE_BF16) for n in numels]
        bc.bc_forecast(h, 0.75, [o.data_ptr() for o in other], bc.DTYPE_BF16, stream())
        for o in outs:
            o.fill_(0)
        torch.cuda.synchronize()
        g.replay()
        torch.cuda.synchronize()
        for a, b in zip(eager, outs):
            assert torch.equal(a, b)
        bc.bc_cache_check(h)
    finally:
        bc.bc_cache_destroy(h)


def test_queued_table_uploads_wait_for_their_staging_buffers():
    # Forecasts over more layers than a parameter block holds upload their layer table through
    # a ring of four pinned staging buffers.  Eight forecasts into eight different output sets,
    # queued behind ~50 ms of device work, need eight uploads: the fifth and later ones must
    # wait until the copies queued earlier have read their staging buffers, and every output
    # set must come out exactly as from a forecast issued alone.
    numels = [(i * 37) % 301 + 1 for i in range(1100)]
    h = run_case(numels, 2, 2, bc.DTYPE_F32, bc.DTYPE_BF16, bc.make_params(), 0.8, [0.9, 0.85],
                 seed=9)
    try:
        ref = [empty_out(n, bc.DTYPE_BF16) for n in numels]
        bc.bc_forecast(h, 0.8, [o.data_ptr() for o in ref], bc.DTYPE_BF16, stream())
        torch.cuda.synchronize()
        sets = [[empty_out(n, bc.DTYPE_BF16) for n in numels] for _ in range(8)]
        st0 = bc.bc_cache_stats(h)
        torch.cuda._sleep(100_000_000)            # device time ahead of the queued uploads
        for outs in sets:
            bc.bc_forecast(h, 0.8, [o.data_ptr() for o in outs], bc.DTYPE_BF16, stream())
        torch.cuda.synchronize()
        assert bc.bc_cache_stats(h)["table_uploads"] - st0["table_uploads"] == 8
        for outs in sets:
            for a, b in zip(ref, outs):
                assert torch.equal(a, b)
        bc.bc_cache_check(h)
    finally:
        bc.bc_cache_destroy(h)


@pytest.mark.parametrize("kernel", KERNELS, ids=KNAME.get)
def test_many_layers_on_two_streams_share_the_device_table(kernel):
    # Forecasts over more layers than a parameter block holds read the handle's one device
    # table.  Issued on two streams without the caller's synchronisation, a call on the other
    # stream must wait for the last launch that read the table: before rewriting it (new
    # outputs) and before reusing the copy queued on that stream.  2048 layers of 32 Ki bf16
    # (512 MiB moved per forecast) keep each launch long enough for a missing wait to show.
    n_l, n = 2048, 32768
    K = 3
    h = bc.bc_cache_create([n] * n_l, K, bc.DTYPE_BF16)
    bc.bc_cache_set_kernel(h, kernel)
    s0 = stream()
    try:
        for j, tau in enumerate((0.9, 0.85, 0.8)):
            slots = bc.bc_cache_next_slot_ptrs(h, n_l)
            offs = bc.bc_cache_layout(h, n_l)
            synth.fill_device(slots[0], bc.DTYPE_BF16, offs[-1] // 2, seed=21, tensor_id=0,
                              step_id=j, tau=tau, degree=2, noise_std=1e-2, stream=s0)
            bc.bc_cache_commit(h, tau)
        t1, t2 = 0.75, 0.7
        ref = {t: [torch.empty(n, dtype=torch.bfloat16, device="cuda") for _ in range(n_l)]
               for t in (t1, t2)}
        for t, outs in ref.items():
            bc.bc_forecast(h, t, [o.data_ptr() for o in outs], bc.DTYPE_BF16, s0)
        torch.cuda.synchronize()
        assert not torch.equal(ref[t1][0], ref[t2][0])
        o1, o2, o3 = ([torch.full((n,), 3.0, dtype=torch.bfloat16, device="cuda")
                       for _ in range(n_l)] for _ in range(3))
        torch.cuda.synchronize()
        sa, sb = torch.cuda.Stream(), torch.cuda.Stream()
        ptr = lambda outs: [o.data_ptr() for o in outs]          # noqa: E731
        st0 = bc.bc_cache_stats(h)
        bc.bc_forecast(h, t1, ptr(o1), bc.DTYPE_BF16, sa.cuda_stream)   # upload on a
        bc.bc_forecast(h, t2, ptr(o2), bc.DTYPE_BF16, sb.cuda_stream)   # rewrite on b
        bc.bc_forecast(h, t2, ptr(o3), bc.DTYPE_BF16, sa.cuda_stream)   # rewrite on a
        bc.bc_forecast(h, t1, ptr(o3), bc.DTYPE_BF16, sb.cuda_stream)   # reuse on b, after a
        torch.cuda.synchronize()
        st1 = bc.bc_cache_stats(h)
        assert st1["table_uploads"] - st0["table_uploads"] == 3
        assert st1["kernel_launches"] - st0["kernel_launches"] == 4
        for got, want in ((o1, ref[t1]), (o2, ref[t2]), (o3, ref[t1])):
            for l in range(n_l):
                assert torch.equal(got[l], want[l]), f"layer {l}"
        bc.bc_cache_check(h)
    finally:
        torch.cuda.synchronize()
        bc.bc_cache_destroy(h)


@pytest.mark.parametrize("kernel", KERNELS, ids=KNAME.get)
def test_many_layer_pushes_on_two_streams_share_the_push_table(kernel):
    # The push table of a cache over 1016 layers, used from two streams: each push on the
    # other stream must wait for the last copy that read the table (new sources rewrite it;
    # reused sources must follow the upload queued on the other stream).  Every slot must
    # hold exactly the bytes of the sources pushed into it.
    n_l, n = 2048, 32768
    h = bc.bc_cache_create([n] * n_l, 3, bc.DTYPE_BF16)
    bc.bc_cache_set_kernel(h, kernel)
    try:
        rng = np.random.default_rng(29)
        srcs = [to_device(rng.integers(0, 2 ** 16, n * n_l, dtype=np.uint16)) for _ in range(3)]
        ptrs = [np.array([s_.data_ptr() + 2 * n * l for l in range(n_l)], dtype=np.uint64)
                for s_ in srcs]
        torch.cuda.synchronize()
        sa, sb = torch.cuda.Stream(), torch.cuda.Stream()
        st0 = bc.bc_cache_stats(h)
        bc.bc_cache_push(h, ptrs[0], 0.9, sa.cuda_stream)     # upload on a
        bc.bc_cache_push(h, ptrs[1], 0.8, sb.cuda_stream)     # rewrite on b
        bc.bc_cache_push(h, ptrs[2], 0.7, sa.cuda_stream)     # rewrite on a
        bc.bc_cache_push(h, ptrs[2], 0.6, sb.cuda_stream)     # reuse on b, after a
        torch.cuda.synchronize()
        bc.bc_cache_check(h)
        st1 = bc.bc_cache_stats(h)
        assert st1["table_uploads"] - st0["table_uploads"] == 3
        assert st1["kernel_launches"] - st0["kernel_launches"] == 4
        assert bc.bc_cache_nodes(h) == [0.6, 0.7, 0.8]
        for j, want in enumerate((srcs[2], srcs[2], srcs[1])):
            slots = bc.bc_cache_slot_ptrs(h, j, n_l)
            for l in range(n_l):
                got = device_view(slots[l], n, bc.DTYPE_BF16)
                assert torch.equal(got, want[l * n:(l + 1) * n]), f"node {j} layer {l}"
    finally:
        torch.cuda.synchronize()
        bc.bc_cache_destroy(h)


@pytest.mark.parametrize("kernel", KERNELS, ids=KNAME.get)
def test_many_layers_with_the_sampler_update(kernel):
    # 1200 layers, the model output among them (index 1100): the fused a x + b v_hat + c z
    # update rides in the one device-table launch; under graph capture the launch is split
    # and the update layer lands in the second parameter-block group.  Both must match the
    # oracle, and the replay the eager result bit for bit.
    numels = [(i * 29) % 513 + 16 for i in range(1200)]
    numels[1100] = 40_000 + 3
    K, times, t_new = 3, [0.9, 0.85, 0.8], 0.75
    feats = synth.host_trajectories([(n,) for n in numels], times, dtype="bf16", seed=41)
    h = bc.bc_cache_create(numels, K, bc.DTYPE_BF16)
    bc.bc_cache_set_kernel(h, kernel)
    try:
        for t, per in zip(times, feats):
            dev = [to_device(f) for f in per]
            bc.bc_cache_push(h, [d.data_ptr() for d in dev], t, stream())
            torch.cuda.synchronize()
        a, b, c = 0.98, -0.05, 0.02
        x0 = np.linspace(-1.0, 1.0, numels[1100]).astype(np.float32)
        z = np.cos(np.arange(numels[1100])).astype(np.float32)
        zd = to_device(z)
        outs = [empty_out(n, bc.DTYPE_BF16) for n in numels]
        for o in outs:
            o.fill_(0)                  # outs[1100] is never written (the update layer)
        ptrs = [o.data_ptr() for o in outs]
        ptrs[1100] = None
        x = to_device(x0)
        l0 = bc.bc_cache_stats(h)["kernel_launches"]
        bc.bc_forecast_update(h, t_new, a, b, c, ptrs, bc.DTYPE_BF16, 1100, x.data_ptr(),
                              bc.DTYPE_F32, zd.data_ptr(), stream())
        torch.cuda.synchronize()
        assert bc.bc_cache_stats(h)["kernel_launches"] - l0 == 1
        W = oracle.paper_weights(times[::-1], t_new)
        nf = feats[::-1]
        x_ref, xb = oracle.update([f[1100] for f in nf], W, x0, a, b, c, z)
        assert_close(to_host(x, bc.DTYPE_F32), x_ref, xb, bc.DTYPE_F32, "x")
        for l in (0, 1099, 1101, 1199):
            ref, bound = oracle.combine([f[l] for f in nf], W)
            assert_close(to_host(outs[l], bc.DTYPE_BF16), ref, bound, bc.DTYPE_BF16, f"layer {l}")
        eager_x = x.clone()
        eager_outs = [o.clone() for o in outs]
        # the same call captured into a graph (parameter-block launches of <= 1016 layers)
        for sel in (1000, 190):                 # first uses of those launchers, uncaptured
            bc.bc_forecast(h, t_new, [q if i < sel else None for i, q in enumerate(ptrs)],
                           bc.DTYPE_BF16, stream())
        x.copy_(to_device(x0))
        torch.cuda.synchronize()
        g = torch.cuda.CUDAGraph()
        s_ = torch.cuda.Stream()
        with torch.cuda.stream(s_):
            with torch.cuda.graph(g, stream=s_, capture_error_mode="thread_local"):
                bc.bc_forecast_update(h, t_new, a, b, c, ptrs, bc.DTYPE_BF16, 1100, x.data_ptr(),
                                      bc.DTYPE_F32, zd.data_ptr(), s_.cuda_stream)
        for o in outs:
            o.fill_(0)
        x.copy_(to_device(x0))
        torch.cuda.synchronize()
        g.replay()
        torch.cuda.synchronize()
        assert torch.equal(x, eager_x)
        for p_, q_ in zip(outs, eager_outs):
            assert torch.equal(p_, q_)
        bc.bc_cache_check(h)
    finally:
        bc.bc_cache_destroy(h)


@pytest.mark.parametrize("in_dt", [bc.DTYPE_BF16, bc.DTYPE_F32])
@pytest.mark.parametrize("K", [1, 2, 3, 4])
def test_small_launch_half_tiles_match_the_register_kernel(in_dt, K):
    # A launch of fewer than two tiles per SM runs the register kernel with half-size tiles
    # under AUTO; pinning REGISTER keeps the full tiles.  Same per-element arithmetic: the
    # outputs must agree bit for bit (and run_case has checked AUTO against the oracle).
    numels = [2 * 256 * 1152, 4097, 13]
    times = [0.9 - 0.05 * i for i in range(K)]
    h = run_case(numels, K, K, in_dt, in_dt, bc.make_params(), times[-1] - 0.05, times,
                 seed=31 + K)
    try:
        res = []
        for kern in (bc.KERNEL_AUTO, bc.KERNEL_REGISTER):
            bc.bc_cache_set_kernel(h, kern)
            outs = [empty_out(n, in_dt) for n in numels]
            bc.bc_forecast(h, times[-1] - 0.05, [o.data_ptr() for o in outs], in_dt, stream())
            torch.cuda.synchronize()
            res.append(outs)
        for a, b in zip(*res):
            assert torch.equal(a, b)
    finally:
        bc.bc_cache_destroy(h)


@pytest.mark.parametrize("kernel", KERNELS, ids=KNAME.get)
@pytest.mark.parametrize("x_dt", [bc.DTYPE_F32, bc.DTYPE_BF16])
@pytest.mark.parametrize("in_dt", [bc.DTYPE_BF16, bc.DTYPE_F32])
@pytest.mark.parametrize("store_v", [False, True])
def test_fused_euler_step(x_dt, in_dt, store_v, kernel):
    numels = [8192 * 2 + 3, 262_144 + 5]   # a block output and a ragged "velocity"
    times = [1.0, 25 / 28, 22 / 28]
    t_new, dt = 21 / 28, -1 / 28
    feats = synth.host_trajectories([(n,) for n in numels], times, dtype=DT_NAME[in_dt], seed=21)
    x0 = synth.host_trajectories([(numels[1],)], [0.0], dtype=DT_NAME[x_dt], degree=0,
                                 noise_std=0.0, seed=22)[0][0]
    h = bc.bc_cache_create(numels, 3, in_dt)
    bc.bc_cache_set_kernel(h, kernel)
    try:
        for t, per in zip(times, feats):
            dev = [to_device(f) for f in per]
            bc.bc_cache_push(h, [d.data_ptr() for d in dev], t, stream())
            torch.cuda.synchronize()
        out0 = empty_out(numels[0], bc.DTYPE_F32)
        vout = empty_out(numels[1], bc.DTYPE_F32) if store_v else None
        x = to_device(x0)
        s0 = bc.bc_cache_stats(h)["kernel_launches"]
        bc.bc_forecast_step(h, t_new, dt, [out0.data_ptr(), vout.data_ptr() if store_v else None],
                            bc.DTYPE_F32, 1, x.data_ptr(), x_dt, stream())
        torch.cuda.synchronize()
        assert bc.bc_cache_stats(h)["kernel_launches"] - s0 == 1
        W = oracle.paper_weights(list(reversed(times)), t_new)
        nf = feats[::-1]
        ref, bound = oracle.combine([f[0] for f in nf], W)
        assert_close(to_host(out0, bc.DTYPE_F32), ref, bound, bc.DTYPE_F32, "block")
        x_ref, v_ref, xb = oracle.euler([f[1] for f in nf], W, x0, dt)
        assert_close(to_host(x, x_dt), x_ref, xb, x_dt, "x")
        if store_v:
            _, vb = oracle.combine([f[1] for f in nf], W)
            assert_close(to_host(vout, bc.DTYPE_F32), v_ref, vb, bc.DTYPE_F32, "v_hat")
    finally:
        bc.bc_cache_destroy(h)


def test_memo_reuses_weights_across_the_schedule():
    # Same differences t - s_j at a later point of an equal-spaced schedule: a memo hit.
    h = bc.bc_cache_create([1024], 2, bc.DTYPE_BF16)
    try:
        z = torch.zeros(1024, dtype=torch.int16, device="cuda")
        bc.bc_cache_push(h, [z.data_ptr()], 0.9, stream())
        bc.bc_cache_push(h, [z.data_ptr()], 0.84, stream())
        c1 = bc.bc_coefficients(h, 0.82)
        bc.bc_cache_push(h, [z.data_ptr()], 0.78, stream())
        c2 = bc.bc_coefficients(h, 0.76)
        torch.cuda.synchronize()
        st = bc.bc_cache_stats(h)
        assert st["memo_misses"] >= 1
        # the differences are (0.02, 0.08) up to rounding of the time grid
        np.testing.assert_allclose(c1, c2, rtol=1e-9)
        c3 = bc.bc_coefficients(h, 0.76)
        assert c3 == c2 and bc.bc_cache_stats(h)["memo_hits"] >= st["memo_hits"] + 1
    finally:
        bc.bc_cache_destroy(h)


def test_empty_layers_and_footprint():
    numels = [0, 5, 0]
    h = bc.bc_cache_create(numels, 2, bc.DTYPE_F32)
    try:
        assert bc.bc_cache_bytes(h) == bc.bc_cache_bytes_for(numels, 2, bc.DTYPE_F32) == 512
        x = torch.arange(5, dtype=torch.float32, device="cuda")
        bc.bc_cache_push(h, [0, x.data_ptr(), 0], 1.0, stream())
        bc.bc_cache_push(h, [0, (x * 2).data_ptr(), 0], 0.5, stream())
        out = torch.empty(5, dtype=torch.float32, device="cuda")
        bc.bc_forecast(h, 0.0, [None, out.data_ptr(), None], bc.DTYPE_F32, stream())
        torch.cuda.synchronize()
        # x(t) = (2 - 2t) * x_base is linear in t: the H = 2 forecast at t = 0 is 2 * x_base
        np.testing.assert_allclose(out.cpu().numpy(), 3.0 * np.arange(5), rtol=1e-6)
    finally:
        bc.bc_cache_destroy(h)
