"""Pins for the fp64 oracle against what the paper and the mathematics fix.

Each pin is chosen so that a plausible slip in ``oracle/oracle.c`` (a dropped term, a wrong
sign or index, a transposed operand, the power applied to the wrong quantity) fails at least
one test.  None of them re-types the oracle's own formula: they use closed forms, textbook
routines (a Vandermonde solve), invariants, limits, and the hand derivations stored in
``tests/golden/coefficients.txt``.
"""
import math
import os

import numpy as np
import pytest

import oracle

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "coefficients.txt")


def _golden_rows():
    rows = []
    with open(GOLDEN) as fh:
        for line in fh:
            line = line.strip()
            if not line or line.startswith("#"):
                continue
            f = [x.strip() for x in line.split(";")]
            name, mode = f[0], f[1]
            nodes = [float(v) for v in f[2].split(",")]
            t = float(f[3])
            num = lambda s: None if s == "-" else float(s)
            rows.append(dict(name=name, mode=mode, nodes=nodes, t=t, delta=num(f[4]),
                             lam=num(f[5]), C=num(f[6]), eta=num(f[7]),
                             W=[float(v) for v in f[8].split(",")]))
    return rows


@pytest.mark.parametrize("row", _golden_rows(), ids=lambda r: r["name"])
def test_golden_coefficients(row):
    if row["mode"] == "exact":
        W = oracle.lagrange(row["nodes"], row["t"])
    else:
        W = oracle.paper_weights(row["nodes"], row["t"], delta=row["delta"], lam=row["lam"],
                                 C=row["C"], eta=row["eta"])
    np.testing.assert_allclose(W, row["W"], rtol=1e-12, atol=1e-12)


# ----------------------------------------------------------------------------- bf16 decode
@pytest.mark.parametrize("bits,value", [
    (0x3F80, 1.0), (0xC000, -2.0), (0x3F81, 1.0 + 2.0 ** -7), (0x4049, 3.140625),
    (0x7F7F, (2.0 - 2.0 ** -7) * 2.0 ** 127), (0x0001, 2.0 ** -133), (0x0080, 2.0 ** -126),
    (0x8000, -0.0), (0x7F80, math.inf), (0xFF80, -math.inf),
])
def test_bf16_decode_known_patterns(bits, value):
    got = float(oracle.bf16_to_float64([bits])[0])
    assert got == value and math.copysign(1.0, got) == math.copysign(1.0, value)


def test_bf16_decode_matches_float32_upper_half():
    rng = np.random.default_rng(7)
    f = rng.standard_normal(4096).astype(np.float32)
    hi = (f.view(np.uint32) >> 16).astype(np.uint16)
    trunc = (hi.astype(np.uint32) << 16).view(np.float32).astype(np.float64)
    np.testing.assert_array_equal(oracle.bf16_to_float64(hi), trunc)


# ------------------------------------------------------------------ exact (Lagrange) weights
@pytest.mark.parametrize("m", [1, 2, 3, 4, 5])
def test_lagrange_matches_vandermonde_solve(m):
    # sum_j c_j s_j^p = t^p for p < m: the defining moment equations, solved by LAPACK.
    rng = np.random.default_rng(100 + m)
    for _ in range(20):
        s = np.sort(rng.uniform(0.0, 1.0, m))[::-1] + np.arange(m)[::-1] * 0.3
        t = s[0] + rng.uniform(0.05, 0.6)
        V = np.vander(s, m, increasing=True).T  # V[p, j] = s_j^p
        rhs = t ** np.arange(m)
        ref = np.linalg.solve(V, rhs)
        np.testing.assert_allclose(oracle.lagrange(s, t), ref, rtol=1e-9, atol=1e-9)


@pytest.mark.parametrize("m", [2, 3, 4])
def test_lagrange_reproduces_polynomials(m):
    rng = np.random.default_rng(200 + m)
    for _ in range(50):
        s = -np.sort(rng.choice(np.arange(0, 1000, 20), m, replace=False)) + 1000.0
        t = float(s.min() - 20 * rng.integers(1, 3))
        s = s / 1000.0
        t = t / 1000.0
        for deg in range(m):
            coef = rng.standard_normal(deg + 1)
            p = np.polynomial.polynomial.polyval
            W = oracle.lagrange(s, t)
            got = float(np.dot(W, p(s, coef)))
            ref = float(p(t, coef))
            scale = float(np.dot(np.abs(W), np.abs(p(s, coef)))) + abs(ref)
            assert abs(got - ref) <= 1e-12 * scale


@pytest.mark.parametrize("K", [1, 2, 3, 4, 5])
def test_lagrange_one_step_past_equispaced_is_binomial(K):
    s = np.arange(K, 0, -1, dtype=np.float64) * 20.0  # newest first, spacing 20
    t = (K + 1) * 20.0
    want = [(-1) ** j * math.comb(K, j + 1) for j in range(K)]
    np.testing.assert_allclose(oracle.lagrange(s, t), want, rtol=1e-13, atol=1e-13)


def test_lagrange_interpolation_property_and_unity():
    s = [0.61, 0.42, 0.27, 0.05]
    for j, sj in enumerate(s):
        np.testing.assert_array_equal(oracle.lagrange(s, sj), np.eye(4)[j])
    rng = np.random.default_rng(3)
    for _ in range(100):
        t = rng.uniform(-1.0, 2.0)
        assert abs(oracle.lagrange(s, t).sum() - 1.0) < 1e-11


def test_lagrange_rejects_duplicate_nodes():
    with pytest.raises(oracle.OracleError):
        oracle.lagrange([0.5, 0.3, 0.5], 0.1)


# -------------------------------------------------------------------- paper weights (Eqs. 8-12)
def test_delta_table_values():
    assert [oracle.delta_table(h) for h in (2, 3, 4)] == [1.0, 0.95, 0.7]


def test_paper_h2_is_linear_extrapolation_for_any_spacing():
    rng = np.random.default_rng(11)
    for _ in range(200):
        s1 = rng.uniform(0.2, 1.0)
        s2 = s1 + rng.uniform(0.06, 0.5)       # older node: larger flow time
        t = s1 - rng.uniform(0.06, 0.4)         # keeps |u| = 0.5/|t-s| below C = 10
        W = oracle.paper_weights([s1, s2], t, delta=1.0, eta=0.0)
        np.testing.assert_allclose(W, oracle.lagrange([s1, s2], t), rtol=1e-12, atol=1e-12)


def test_paper_h3_equispaced_is_quadratic_extrapolation():
    for h in (20.0, 1.0 / 28, 0.05):
        for steps in (1, 2, 3):
            s = [3 * h, 4 * h, 5 * h]
            t = 3 * h - steps * h
            W = oracle.paper_weights(s, t, delta=1.0, eta=0.0, C=1e30)
            np.testing.assert_allclose(W, oracle.lagrange(s, t), rtol=1e-11, atol=1e-11)


@pytest.mark.parametrize("H", [2, 3, 4, 5, 6])
def test_paper_reproduces_lines_on_equispaced_nodes(H):
    # Floater-Hormann with d = 1 reproduces linear functions (remark under Eq. 8).
    s = np.arange(H, dtype=np.float64)[::-1] + 1.0  # H, ..., 1 (newest first)
    for t in (H + 0.5, H + 1.0, H + 3.0, 0.25, -2.0):
        W = oracle.paper_weights(s, t, delta=1.0, eta=0.0, C=1e30)
        assert abs(W.sum() - 1.0) < 1e-12
        assert abs(float(np.dot(W, s)) - t) < 1e-11 * (1 + abs(t))


def test_paper_reuse_and_unity():
    rng = np.random.default_rng(5)
    for _ in range(200):
        H = int(rng.integers(1, 5))
        s = np.sort(rng.uniform(0, 1, H))
        t = float(s[0] - rng.uniform(0.001, 0.3))
        lam = float(rng.uniform(0, 1))
        W = oracle.paper_weights(s, t, lam=lam)
        assert abs(W.sum() - 1.0) < 1e-12
        W1 = oracle.paper_weights(s, t, lam=1.0)
        np.testing.assert_allclose(W1, np.eye(H)[0], atol=1e-15)


def test_paper_translation_invariance():
    # Weights depend only on the differences t - s_j (the Diff Key argument, Eq. 7).
    s = np.array([740.0, 760.0, 800.0, 860.0])
    for shift in (-512.0, 0.0, 256.0, 4096.0):
        a = oracle.paper_weights(s, 720.0)
        b = oracle.paper_weights(s + shift, 720.0 + shift)
        np.testing.assert_allclose(a, b, rtol=1e-13, atol=1e-13)


@pytest.mark.parametrize("delta", [0.3, 0.7, 0.95, 1.0])
def test_paper_scale_invariance_without_clip(delta):
    # Scaling every t - s_j by k scales each |u_j| by 1/k and each a_j by k^-delta: alpha
    # is unchanged if the power is applied to every |u~_j| alike (eta = 0, no clip).
    s = np.array([0.30, 0.45, 0.55, 0.80])
    t = 0.10
    a = oracle.paper_weights(s, t, delta=delta, eta=0.0, C=1e30)
    for k in (0.25, 2.0, 8.0):
        b = oracle.paper_weights(s * k, t * k, delta=delta, eta=0.0, C=1e30)
        np.testing.assert_allclose(a, b, rtol=1e-12, atol=1e-12)


def test_paper_small_delta_limit_is_sign_average():
    # delta -> 0: a_j -> sgn(u~_j), so alpha_j -> sgn_j / sum sgn.  With the alternating
    # signs of Eq. 9 and three nodes that is (+1, -1, +1) / 1.
    W = oracle.paper_weights([0.5, 0.6, 0.7], 0.45, delta=1e-9, eta=0.0)
    np.testing.assert_allclose(W, [1.0, -1.0, 1.0], atol=1e-7)


def test_paper_alternating_signs_follow_eq9():
    # Target beyond every node: all t - s_j share one sign, so Eq. 9's (-1)^j alternates u_j.
    W = oracle.paper_weights([0.5, 0.6, 0.7, 0.8], 0.45, delta=0.7, eta=1e-12)
    assert list(np.sign(W)) == [1.0, -1.0, 1.0, -1.0]


def test_paper_clip_bounds_node_hit():
    # t equal to a node: Eq. 9 divides by t - s_1 = +0, so u_1 = c_1 (-1)^1 / +0 = -inf and
    # Eq. 10 clips it to -C.  The result is finite, sums to one, and equals the one-sided limit
    # from t > s_1 (where t - s_1 is also positive and u_1 is clipped to -C as well).  From the
    # other side u_1 has the opposite sign, so the two one-sided limits differ.
    s = [0.5, 0.6, 0.7]
    W_hit = oracle.paper_weights(s, 0.5)
    W_above = oracle.paper_weights(s, 0.5 + 1e-9)
    W_below = oracle.paper_weights(s, 0.5 - 1e-9)
    assert np.all(np.isfinite(W_hit)) and abs(W_hit.sum() - 1.0) < 1e-12
    np.testing.assert_allclose(W_hit, W_above, rtol=1e-7, atol=1e-7)
    assert np.max(np.abs(W_below - W_hit)) > 1.0


def test_paper_clip_equals_substituting_c():
    # Whenever |u_1| exceeds C the weights must equal those of a target where u_1 = -+C exactly
    # and the other u_j are unchanged: move only the first node so that 0.5/|t - s_1| = C.
    s = [0.78, 0.9, 1.0]
    t = 0.76                       # u_1 = 0.5/0.02 = 25 -> clipped to 10
    W_clip = oracle.paper_weights(s, t, delta=1.0, eta=0.0)
    s_sub = [t + 0.05, 0.9, 1.0]   # u_1 = -0.5/(t - s_1) = 0.5/0.05 = 10 exactly
    np.testing.assert_allclose(W_clip, oracle.paper_weights(s_sub, t, delta=1.0, eta=0.0),
                               rtol=1e-12)


def test_paper_degenerate_normalisation_is_reported():
    # H = 2, both raw weights clipped to +-C with opposite signs: sum a_j = 0.
    with pytest.raises(oracle.OracleError):
        oracle.paper_weights([0.01, 0.02], 0.0, delta=1.0, eta=0.0)


# ------------------------------------------------------------------- Eq. 13 combination pins
def _poly_nodes_data(dtype, m, n, seed):
    # Integer-valued polynomials of degree m-1 at integer nodes: every stored value is exact
    # in fp32 (< 2^24) and, for the bf16 case, in bf16 (|v| < 256 integers).
    rng = np.random.default_rng(seed)
    s = np.arange(m, dtype=np.float64)[::-1] * 1.0 + 1.0   # m..1, newest first
    t = float(m + 1)
    lim = 2 if dtype == "bf16" else 50
    coef = rng.integers(-lim, lim + 1, size=(m, n)).astype(np.float64)
    vals = [sum(coef[d] * sj ** d for d in range(m)) for sj in s]
    want = sum(coef[d] * t ** d for d in range(m))
    if dtype == "bf16":
        assert max(np.abs(v).max() for v in vals) < 256
        F = [(v.astype(np.float32).view(np.uint32) >> 16).astype(np.uint16) for v in vals]
    else:
        F = [v.astype(np.float32) for v in vals]
    return s, t, F, want


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
@pytest.mark.parametrize("m", [1, 2, 3, 4])
def test_combine_reproduces_polynomial_data(dtype, m):
    s, t, F, want = _poly_nodes_data(dtype, m, 1031, seed=m)
    W = oracle.lagrange(s, t)
    got, bound = oracle.combine(F, W)
    assert np.all(np.abs(got - want) <= 1e-12 * (bound + 1.0))


def test_combine_bound_is_weighted_magnitude():
    F = [np.full(5, 2.0, np.float32), np.full(5, -3.0, np.float32)]
    out, bound = oracle.combine(F, [0.5, -0.25])
    np.testing.assert_array_equal(out, np.full(5, 1.75))
    np.testing.assert_array_equal(bound, np.full(5, 1.75))
    out, bound = oracle.combine(F, [0.5, 0.25])
    np.testing.assert_array_equal(out, np.full(5, 0.25))
    np.testing.assert_array_equal(bound, np.full(5, 1.75))


def test_combine_node_order_matters():
    # A transposed node order would pair W_1 with the oldest tensor.
    F = [np.arange(4, dtype=np.float32), np.zeros(4, np.float32)]
    out, _ = oracle.combine(F, [2.0, -1.0])
    np.testing.assert_array_equal(out, 2.0 * np.arange(4))


def test_euler_on_linear_velocity():
    # Velocity linear in t, sampled at three equispaced flow times; the forecast at t is exact
    # and the Euler step adds dt * v(t): x' = x + dt (a + b t).
    rng = np.random.default_rng(9)
    n = 257
    a = rng.integers(-8, 9, n).astype(np.float64)
    b = rng.integers(-8, 9, n).astype(np.float64)
    s = [0.75, 0.875, 1.0]
    t, dt = 0.625, -0.125
    V = [(a + b * sj).astype(np.float32) for sj in s]
    x = rng.integers(-100, 100, n).astype(np.float32)
    W = oracle.lagrange(s, t)
    x_new, v_hat, bound = oracle.euler(V, W, x, dt)
    np.testing.assert_allclose(v_hat, a + b * t, atol=1e-12)
    np.testing.assert_allclose(x_new, x + dt * (a + b * t), atol=1e-12)
    assert np.all(bound >= np.abs(x))
