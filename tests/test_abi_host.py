"""Host-side checks of the C-ABI library that need no GPU.

* the library loads and exports every entry point ``include/barycache.h`` declares;
* the host fp64 solver (second barycentric form / Eqs. 8-12 from differences) agrees with
  the oracle's independent Lagrange-product and step-by-step implementations;
* footprints, status strings, argument validation and the schedule arithmetic.
"""
import ctypes
import math
import os
import re

import numpy as np
import pytest

import oracle
from paper_2608_28670_gb300 import barycache as bc
from paper_2608_28670_gb300 import synth
from paper_2608_28670_gb300.configs import WORKLOADS, T2V_HBM_BUDGET

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "barycache.h")


@pytest.fixture(scope="module", autouse=True)
def built():
    import __graft_entry__
    __graft_entry__.build_libraries()


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(bc_[a-z_]+)\s*\(", text)))


def test_every_declared_symbol_is_exported():
    names = declared_functions()
    assert len(names) >= 20
    L = ctypes.CDLL(bc.LIB_PATH)
    for n in names:
        assert hasattr(L, n), n
    assert sorted(bc.exported_names()) == names


def test_version_and_status_strings():
    assert bc.bc_version() >= 10000
    L = bc.lib()
    seen = set()
    for s in range(10):
        msg = L.bc_status_string(s).decode()
        assert msg and msg not in seen
        seen.add(msg)
    assert L.bc_status_string(1234).decode() == "unknown status"


def test_default_params_are_the_papers():
    p = bc.bc_params_default()
    assert (p.mode, p.delta, p.lambda_, p.clip_C, p.eta) == (bc.MODE_PAPER, 0.0, 0.0, 10.0, 1e-12)


# ------------------------------------------------------------------- solver vs oracle
def _random_window(rng, m, kind):
    if kind == "ddim":
        steps = rng.choice(np.arange(1, 49), m, replace=False)
        nodes = np.sort(980.0 - 20.0 * steps)   # time runs down: newest = smallest t
        t = float(nodes[0] - 20.0 * rng.integers(1, 3))
    else:
        nodes = np.sort(rng.choice(np.arange(1, 49), m, replace=False) / 50.0)
        t = float(nodes[0] - rng.integers(1, 3) / 50.0)
    return nodes, t


@pytest.mark.parametrize("m", [1, 2, 3, 4])
@pytest.mark.parametrize("kind", ["ddim", "flow"])
def test_exact_mode_matches_oracle_lagrange(m, kind):
    rng = np.random.default_rng(m * 7 + len(kind))
    prm = bc.make_params(mode=bc.MODE_EXACT)
    for _ in range(100):
        nodes, t = _random_window(rng, m, kind)
        got = np.array(bc.bc_solve(nodes, t, prm))
        ref = oracle.lagrange(nodes, t)
        np.testing.assert_allclose(got, ref, rtol=1e-10, atol=1e-10 * np.abs(ref).max())


@pytest.mark.parametrize("m", [1, 2, 3, 4])
@pytest.mark.parametrize("kind", ["ddim", "flow"])
@pytest.mark.parametrize("lam", [0.0, 0.3, 1.0])
def test_paper_mode_matches_oracle(m, kind, lam):
    rng = np.random.default_rng(m * 13 + int(lam * 10))
    prm = bc.make_params(mode=bc.MODE_PAPER, lam=lam)
    for _ in range(100):
        nodes, t = _random_window(rng, m, kind)
        try:
            ref = oracle.paper_weights(nodes, t, lam=lam)
        except oracle.OracleError:
            with pytest.raises(bc.BaryCacheError) as ei:
                bc.bc_solve(nodes, t, prm)
            assert ei.value.status == bc.ERR_DEGENERATE_WEIGHTS
            continue
        got = np.array(bc.bc_solve(nodes, t, prm))
        np.testing.assert_allclose(got, ref, rtol=1e-12, atol=1e-12)


def test_paper_mode_explicit_delta_and_clip():
    prm = bc.make_params(mode=bc.MODE_PAPER, delta=0.5, clip_C=3.0, eta=0.0)
    nodes, t = [0.55, 0.7, 0.85, 1.0], 0.5
    np.testing.assert_allclose(bc.bc_solve(nodes, t, prm),
                               oracle.paper_weights(nodes, t, delta=0.5, C=3.0, eta=0.0),
                               rtol=1e-12, atol=1e-12)


def test_node_hit_behaviour():
    nodes = [0.5, 0.6, 0.7]
    np.testing.assert_array_equal(bc.bc_solve(nodes, 0.6, bc.make_params(mode=bc.MODE_EXACT)),
                                  [0.0, 1.0, 0.0])
    np.testing.assert_allclose(bc.bc_solve(nodes, 0.5), oracle.paper_weights(nodes, 0.5),
                               rtol=1e-12)


@pytest.mark.parametrize("nodes,t,params,status", [
    ([0.5, 0.5], 0.4, dict(mode=0), bc.ERR_DUPLICATE_NODE),
    ([0.01, 0.02], 0.0, dict(delta=1.0, eta=0.0), bc.ERR_DEGENERATE_WEIGHTS),
    ([0.5], float("nan"), dict(), bc.ERR_INVALID_ARG),
    ([0.5, float("inf")], 0.4, dict(), bc.ERR_INVALID_ARG),
    ([0.5, 0.6], 0.4, dict(lam=1.5), bc.ERR_INVALID_ARG),
    ([0.5, 0.6], 0.4, dict(clip_C=0.0), bc.ERR_INVALID_ARG),
    ([0.5, 0.6], 0.4, dict(eta=-1.0), bc.ERR_INVALID_ARG),
    ([0.5, 0.6], 0.4, dict(mode=7), bc.ERR_INVALID_ARG),
    ([0.1, 0.2, 0.3, 0.4, 0.5], 0.0, dict(), bc.ERR_INVALID_ARG),
])
def test_solver_errors(nodes, t, params, status):
    with pytest.raises(bc.BaryCacheError) as ei:
        bc.bc_solve(nodes, t, bc.make_params(**params))
    assert ei.value.status == status
    assert bc.lib().bc_last_error().decode()


def test_solver_rejects_empty_window():
    with pytest.raises(bc.BaryCacheError) as ei:
        bc.bc_solve([], 0.3)
    assert ei.value.status == bc.ERR_INVALID_ARG


# ------------------------------------------------------------------- footprint
def test_footprints_of_the_five_workloads():
    # K slots x sum of 256-byte aligned layer sizes (every size here is already aligned).
    want = {"c2i-256": 7_077_888, "c2i-512": 2_113_929_216, "t2i-1024": 3_170_893_824}
    for name, b in want.items():
        w = WORKLOADS[name]
        assert bc.bc_cache_bytes_for(w.numels, w.K, w.dtype) == b == w.cache_bytes()
    w = WORKLOADS["mmdit-t2i"]
    assert bc.bc_cache_bytes_for(w.numels, w.K, w.dtype) == 4_841_275_392 + 3 * 524_288
    w = WORKLOADS["t2v"]
    got = [bc.bc_cache_bytes_for(w.numels, K, w.dtype) for K in (2, 3, 4)]
    assert got == [87_588_864_000, 131_383_296_000, 175_177_728_000]
    # What fits the stated 180 GB budget together with a full-size forecast output.
    out = w.layer_numel * w.n_layers * 2
    assert [g + out <= T2V_HBM_BUDGET for g in got] == [True, True, False]


def test_footprint_alignment_and_validation():
    assert bc.bc_cache_bytes_for([1], 1, bc.DTYPE_BF16) == 256
    assert bc.bc_cache_bytes_for([129, 0, 64], 2, bc.DTYPE_F32) == 2 * (768 + 0 + 256)
    for args in [([], 1, 0), ([10], 0, 0), ([10], 5, 0), ([10], 1, 3), ([-1], 1, 0)]:
        with pytest.raises(bc.BaryCacheError) as ei:
            bc.bc_cache_bytes_for(*args)
        assert ei.value.status == bc.ERR_INVALID_ARG


def test_create_without_a_device_fails_loudly():
    import torch
    if torch.cuda.is_available():
        pytest.skip("a device is present")
    with pytest.raises(bc.BaryCacheError) as ei:
        bc.bc_cache_create([16], 2, bc.DTYPE_BF16)
    assert ei.value.status == bc.ERR_CUDA


def test_calls_on_a_null_handle():
    for fn, args in [(bc.bc_cache_bytes, ()), (bc.bc_cache_nodes, ()), (bc.bc_cache_reset, ()),
                     (bc.bc_coefficients, (0.5,)), (bc.bc_cache_commit, (0.5,)),
                     (bc.bc_cache_stats, ()), (bc.bc_cache_destroy, ())]:
        with pytest.raises(bc.BaryCacheError) as ei:
            fn(0, *args)
        assert ei.value.status == bc.ERR_BAD_HANDLE


# ------------------------------------------------------------------- schedules
def test_schedule_full_step_counts_match_the_flops_tables():
    # Tables 1 and 3: FLOPs(BaryCache) / FLOPs(one vanilla step) = number of full steps.
    # 126.15 / (450.52 / 50) = 14.0 (N=4), 90.10 / 9.0104 = 10.0 (N=6)  [Table 1, H = 2]
    # 5.24 / (23.74 / 50) = 11.04 (N=5), 4.77 / 0.4748 = 10.05 (N=6)    [Table 3, H = 2]
    from dataclasses import replace
    base = WORKLOADS["c2i-512"]
    for interval, flops, vanilla in [(4, 126.15, 450.52), (6, 90.10, 450.52),
                                     (5, 5.24, 23.74), (6, 4.77, 23.74)]:
        w = replace(base, interval=interval, K=2)
        full = sum(w.is_full(i) for i in range(50))
        assert full == math.ceil(50 / interval) + 1
        assert abs(flops / (vanilla / 50) - full) < 0.1


def test_representative_problems():
    w = WORKLOADS["c2i-512"]
    p = w.representative()
    assert p.nodes == (500.0, 560.0, 620.0, 680.0) and p.t == 480.0
    t2v = WORKLOADS["t2v"]
    fc = [p.step for p in t2v.problems()]
    assert all(not t2v.is_full(i) for i in fc)
    # forecasting two of every three steps once the window is full
    assert all((s % 3) in (1, 2) for s in fc)
    for K in (2, 3, 4):
        p = t2v.representative(K)
        assert len(p.nodes) == K and p.nodes[0] > p.t


def test_host_bf16_rounding_is_nearest_even():
    f = np.array([1.0, 1.0 + 2 ** -8, 1.0 + 3 * 2 ** -8, -2.5, 3.0e38], dtype=np.float32)
    bits = synth.f32_to_bf16_bits(f)
    assert list(bits[:3]) == [0x3F80, 0x3F80, 0x3F82]
    np.testing.assert_array_equal(synth.bf16_bits_to_f32(bits)[3], np.float32(-2.5))


# ------------------------------------------------------------------- sampler coefficients
@pytest.mark.parametrize("alpha_t,alpha_bar_t", [(0.9999, 0.9999), (0.98, 0.5), (0.99, 1e-4),
                                                  (1.0, 0.3)])
def test_ddpm_coefficients_match_oracle(alpha_t, alpha_bar_t):
    np.testing.assert_allclose(bc.bc_ddpm_coefficients(alpha_t, alpha_bar_t),
                               oracle.ddpm_coefficients(alpha_t, alpha_bar_t), rtol=1e-14)


@pytest.mark.parametrize("ab_t,ab_prev,eta", [(0.1, 0.2, 0.0), (0.1, 0.2, 1.0), (0.5, 0.9, 0.5),
                                              (0.999, 1.0, 0.0), (1e-3, 0.05, 0.3)])
def test_ddim_coefficients_match_oracle(ab_t, ab_prev, eta):
    np.testing.assert_allclose(bc.bc_ddim_coefficients(ab_t, ab_prev, eta),
                               oracle.ddim_coefficients(ab_t, ab_prev, eta), rtol=1e-13,
                               atol=1e-15)


def test_sampler_coefficient_errors():
    for args in [(0.0, 0.5), (0.9, 1.0)]:
        with pytest.raises(bc.BaryCacheError):
            bc.bc_ddpm_coefficients(*args)
    for args in [(0.5, 0.4, 0.0), (0.5, 0.6, -1.0), (0.1, 0.9, 5.0)]:
        with pytest.raises(bc.BaryCacheError):
            bc.bc_ddim_coefficients(*args)


# ------------------------------------------------------------------- schedules
def test_equal_schedule_matches_the_flops_tables_and_configs():
    for interval, full in [(4, 14), (5, 11), (6, 10)]:      # Tables 1 and 3, H = 2
        assert sum(bc.bc_schedule_equal(50, interval, 2)) == full
    for name in ("c2i-512", "t2i-1024", "mmdit-t2i", "t2v"):
        w = WORKLOADS[name]
        assert bc.bc_schedule_equal(w.steps, w.interval, w.K) == \
            [int(w.is_full(i)) for i in range(w.steps)]
    assert bc.bc_schedule_equal(0, 3, 2) == []
    with pytest.raises(bc.BaryCacheError):
        bc.bc_schedule_equal(10, 0, 2)


def test_adaptive_schedule_accumulates_and_resets():
    st = bc.bc_adaptive_init(0.25, 2)
    drifts = [0.0, 0.3, 0.1, 0.1, 0.06, 0.2, 0.01, 0.5, 0.0]
    # steps 0, 1: window fills (full); then 0.1, 0.2 (skip), 0.26 >= 0.25 (full, reset),
    # 0.2 (skip), 0.21 (skip), 0.71 (full, reset), 0.0 (skip)
    want = [1, 1, 0, 0, 1, 0, 0, 1, 0]
    assert [bc.bc_adaptive_decide(st, d) for d in drifts] == want
    assert st.full_steps == 4 and st.steps == 9 and st.accumulated == 0.0
    st0 = bc.bc_adaptive_init(0.0, 0)              # threshold 0: every step is full
    assert all(bc.bc_adaptive_decide(st0, 0.0) for _ in range(5))
    with pytest.raises(bc.BaryCacheError):
        bc.bc_adaptive_decide(st, float("nan"))
    with pytest.raises(bc.BaryCacheError):
        bc.bc_adaptive_init(-1.0, 2)


def test_pointer_tables_from_lists_and_numpy_arrays():
    # Both forms reach C as the same array of addresses (None / 0 = NULL); numpy tables are
    # passed without a per-element conversion.
    addrs = [16, None, 2 ** 40 + 32, 0]
    want = [16, None, 2 ** 40 + 32, None]
    p = bc._ptr_array(addrs)
    assert [p[i] for i in range(4)] == want
    for dt in (np.uint64, np.int64):
        a = np.array([q or 0 for q in addrs], dtype=dt)
        p = bc._ptr_array(a)
        assert [p[i] for i in range(4)] == want
    with pytest.raises(TypeError):
        bc._ptr_array(np.array([16, 32], dtype=np.uint32))
    with pytest.raises(TypeError):
        bc._ptr_array(np.zeros((2, 2), dtype=np.uint64))


def _golden():
    from tests.test_oracle_pins import _golden_rows
    return _golden_rows()


@pytest.mark.parametrize("row", _golden(), ids=lambda r: r["name"])
def test_library_solver_matches_the_hand_derived_weights(row):
    # The library's own fp64 solver (not just the oracle) against the worked examples.
    if row["mode"] == "exact":
        prm = bc.make_params(mode=bc.MODE_EXACT)
    else:
        prm = bc.make_params(mode=bc.MODE_PAPER, delta=row["delta"], lam=row["lam"],
                             clip_C=row["C"], eta=row["eta"])
    got = bc.bc_solve(row["nodes"], row["t"], prm)
    np.testing.assert_allclose(got, row["W"], rtol=1e-12, atol=1e-12)
