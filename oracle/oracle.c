/*
 * oracle.c -- plain, slow, fp64 CPU oracle for the BaryCache skipped-step forecast.
 *
 * TEST INFRASTRUCTURE ONLY.  Nothing in the product path may link, load or call this
 * file.  It is used by the tests, by the smoke check and by the CPU-baseline leg of the
 * benchmark, and by nothing else.  It shares no code, header, table or constant with the
 * CUDA library: every formula below is written out again from the paper.
 *
 * What it computes (BaryCache, "Barycentric Extrapolator", Sec. 3.2 and 3.3):
 *   - the exact polynomial extrapolation coefficients in the explicit Lagrange form
 *     (the classical definition that barycentric interpolation re-expresses; Sec. 1 and
 *     the remark under Eq. 8);
 *   - the paper's stabilised weights, Eqs. 8-12, step by step in the paper's order;
 *   - the weight application of Eq. 13, x_hat = sum_j W_j * x_{f=-j}, element by element;
 *   - the fused Euler update x <- x + dt * x_hat used by the flow-matching sampler (Sec. 4.1);
 *   - the DDPM step of Eqs. 2-3, the DDIM step (from the DDIM paper; the sampler the paper
 *     uses for C2I/T2I, Sec. 4.1) and the general update x <- a x + b x_hat + c z;
 *   - the relative L1 drift of a feature probe that drives the adaptive schedule (Sec. 4.5).
 *
 * Index convention (Sec. 3.2, "Get Key"): node j = 1 is the most recent cached feature
 * x_{f=-1} with timestep s_1; node H is the oldest.  In C arrays that is index j-1.
 *
 * Everything is evaluated in double precision.  Stored inputs (fp32 or bf16) convert to
 * double exactly, so the oracle's result is the mathematically defined value up to fp64
 * rounding.
 *
 * Pins (tests/test_oracle_pins.py, tests/test_oracle_samplers.py): every function is checked
 * against closed forms, identities or library routines.  For the paper's weights with a decay
 * power delta != 1 the paper prints no value; they are pinned by hand-derived closed forms at
 * delta = 2 and 1/2 (where the powers are exact: squares and square roots, including a case
 * with the clip active) and by invariants and limits (scale invariance, the delta -> 0 limit,
 * sign alternation, unit sum, translation invariance).
 */
#include <math.h>
#include <stdint.h>
#include <string.h>

#define ORACLE_OK 0
#define ORACLE_DUPLICATE_NODE 1
#define ORACLE_DEGENERATE 2
#define ORACLE_BAD_ARG 3

#define ORACLE_F32 0
#define ORACLE_BF16 1

/* ---------------------------------------------------------------------------------
 * Stored-value decoding.  A bf16 value is the upper half of an IEEE-754 binary32
 * word; widening it is a 16-bit left shift, which is exact.
 * ------------------------------------------------------------------------------- */
double oracle_bf16_to_double(uint16_t bits)
{
    uint32_t word = ((uint32_t)bits) << 16;
    float f;
    memcpy(&f, &word, sizeof f);
    return (double)f;
}

static double load_elem(int dtype, const void *base, int64_t e)
{
    if (dtype == ORACLE_BF16) {
        const uint16_t *p = (const uint16_t *)base;
        return oracle_bf16_to_double(p[e]);
    } else {
        const float *p = (const float *)base;
        return (double)p[e];
    }
}

/* ---------------------------------------------------------------------------------
 * Exact extrapolation coefficients, explicit Lagrange form.
 *
 *   c_j = prod_{k != j} (t - s_k) / (s_j - s_k),   j = 1..m
 *
 * This is the polynomial of degree m-1 through the m cached nodes evaluated at the
 * target t; the barycentric formula c_j = (w_j/(t-s_j)) / sum_k (w_k/(t-s_k)) with
 * w_j = 1/prod_{k!=j}(s_j - s_k) is the same number written differently.  At t == s_j
 * the product form gives e_j directly, with no special case.
 * Returns ORACLE_DUPLICATE_NODE if two nodes coincide (the polynomial is undefined).
 * ------------------------------------------------------------------------------- */
int oracle_lagrange(const double *s, int m, double t, double *c)
{
    if (m < 1) return ORACLE_BAD_ARG;
    for (int j = 0; j < m; ++j)
        for (int k = j + 1; k < m; ++k)
            if (s[j] == s[k]) return ORACLE_DUPLICATE_NODE;
    for (int j = 0; j < m; ++j) {
        double prod = 1.0;
        for (int k = 0; k < m; ++k) {
            if (k == j) continue;
            prod *= (t - s[k]) / (s[j] - s[k]);
        }
        c[j] = prod;
    }
    return ORACLE_OK;
}

/* Decay factor delta_H chosen empirically in Sec. 3.2 (text under Eq. 10):
 * 1.0 for H = 2, 0.95 for H = 3, 0.7 for H = 4.  A one-node window (H = 1) has a
 * single weight that normalises to 1 whatever delta is; 1.0 is returned for it.
 * Other H are not given by the paper: returns a negative number. */
double oracle_delta_table(int H)
{
    switch (H) {
    case 1: return 1.0;
    case 2: return 1.0;
    case 3: return 0.95;
    case 4: return 0.7;
    default: return -1.0;
    }
}

static double sgn_plus(double v) { return v < 0.0 ? -1.0 : 1.0; } /* sgn(0) := +1 */

/* ---------------------------------------------------------------------------------
 * The paper's weights, Eqs. 8-12, in the paper's order.
 *
 *   Eq. 8   trapezoid-like node factors: c_1 = c_H = 0.5, c_j = 1 for 2 <= j <= H-1
 *   Eq. 9   raw weight   u_j = c_j (-1)^j / (t - s_j)
 *   Eq. 10  clip         u~_j = max(-C, min(C, u_j))
 *   Eq. 11  decay power  a_j = sgn(u~_j) (|u~_j| + eta)^delta,  alpha_j = a_j / sum_m a_m
 *   Eq. 12  blend        W = (1 - lambda) alpha + lambda e_1
 *
 * Eq. 12 as printed scales the first H-1 entries by (1-lambda) and the last by lambda;
 * the text says the blend mixes the extrapolation with the most recent feature x_{f=-1}.
 * This oracle follows the text: W_1 gains lambda, every alpha_j is scaled by (1-lambda),
 * so sum W = 1, lambda = 0 is pure extrapolation and lambda = 1 is reuse of x_{f=-1}.
 *
 * At t == s_j the IEEE division gives +-inf, which the clip maps to +-C.
 * Returns ORACLE_DEGENERATE when |sum_m a_m| < 1e-12 * sum_m |a_m| (no usable
 * normalisation; the paper does not cover this case).
 * ------------------------------------------------------------------------------- */
int oracle_paper_weights(const double *s, int m, double t, double delta, double lambda,
                         double C, double eta, double *W)
{
    double cfac[64], u[64], ut[64], a[64];
    if (m < 1 || m > 64 || !(C > 0.0) || !(delta > 0.0) || eta < 0.0) return ORACLE_BAD_ARG;

    /* Eq. 8 */
    for (int j = 1; j <= m; ++j) cfac[j - 1] = (j == 1 || j == m) ? 0.5 : 1.0;

    /* Eq. 9: (-1)^j with j counted from 1 */
    for (int j = 1; j <= m; ++j) {
        double sign = (j % 2 == 0) ? 1.0 : -1.0;
        u[j - 1] = cfac[j - 1] * sign / (t - s[j - 1]);
    }

    /* Eq. 10 */
    for (int j = 0; j < m; ++j) ut[j] = fmax(-C, fmin(C, u[j]));

    /* Eq. 11 */
    double sum = 0.0, sum_abs = 0.0;
    for (int j = 0; j < m; ++j) {
        a[j] = sgn_plus(ut[j]) * pow(fabs(ut[j]) + eta, delta);
        sum += a[j];
        sum_abs += fabs(a[j]);
    }
    if (!(fabs(sum) >= 1e-12 * sum_abs) || sum_abs == 0.0) return ORACLE_DEGENERATE;

    /* Eq. 11 normalisation followed by the Eq. 12 blend towards x_{f=-1} */
    for (int j = 0; j < m; ++j) {
        double alpha = a[j] / sum;
        W[j] = (1.0 - lambda) * alpha + (j == 0 ? lambda : 0.0);
    }
    return ORACLE_OK;
}

/* ---------------------------------------------------------------------------------
 * Eq. 13: x_hat[e] = sum_{j=1..m} W_j * F_j[e], in fp64 from the stored values.
 * F[j] points to the stored tensor of node j (j = 0 is x_{f=-1}), each holding n
 * elements of `dtype`.  Also returns bound[e] = sum_j |W_j| |F_j[e]|, the scale that the
 * per-element tolerance is measured against.  `bound` may be NULL.
 * ------------------------------------------------------------------------------- */
void oracle_combine(int dtype, const void *const *F, int m, const double *W, int64_t n,
                    double *out, double *bound)
{
    for (int64_t e = 0; e < n; ++e) {
        double acc = 0.0, mag = 0.0;
        for (int j = 0; j < m; ++j) {
            double v = load_elem(dtype, F[j], e);
            acc += W[j] * v;
            mag += fabs(W[j]) * fabs(v);
        }
        out[e] = acc;
        if (bound) bound[e] = mag;
    }
}

/* ---------------------------------------------------------------------------------
 * Forecast followed by one explicit Euler step of the flow-matching sampler:
 *   v_hat[e] = sum_j W_j V_j[e]          (Eq. 13 applied to the cached velocity)
 *   x_out[e] = x[e] + dt * v_hat[e]
 * x is stored in x_dtype.  v_hat may be NULL.  bound[e] = |x[e]| + |dt| sum_j |W_j||V_j[e]|.
 * ------------------------------------------------------------------------------- */
void oracle_euler(int v_dtype, const void *const *V, int m, const double *W, int64_t n,
                  double dt, int x_dtype, const void *x, double *x_out, double *v_hat,
                  double *bound)
{
    for (int64_t e = 0; e < n; ++e) {
        double acc = 0.0, mag = 0.0;
        for (int j = 0; j < m; ++j) {
            double v = load_elem(v_dtype, V[j], e);
            acc += W[j] * v;
            mag += fabs(W[j]) * fabs(v);
        }
        double x0 = load_elem(x_dtype, x, e);
        x_out[e] = x0 + dt * acc;
        if (v_hat) v_hat[e] = acc;
        if (bound) bound[e] = fabs(x0) + fabs(dt) * mag;
    }
}

/* ---------------------------------------------------------------------------------
 * Sampler updates applied to the forecast of the cached model output.
 *
 * DDPM reverse step, Sec. 3.1: Eq. 3 gives the mean
 *     mu = (1 / sqrt(alpha_t)) * (x_t - (1 - alpha_t) / sqrt(1 - alpha_bar_t) * eps)
 * and Eq. 2 the variance beta_t; beta_t is read as 1 - alpha_t, the noise variance of the
 * forward step in Eq. 1.  Written as x_{t-1} = a x_t + b eps + c z.
 * ------------------------------------------------------------------------------- */
int oracle_ddpm_coefficients(double alpha_t, double alpha_bar_t, double *a, double *b,
                             double *c)
{
    if (!(alpha_t > 0.0 && alpha_t <= 1.0) || !(alpha_bar_t > 0.0 && alpha_bar_t < 1.0))
        return ORACLE_BAD_ARG;
    double inv_sqrt_alpha = 1.0 / sqrt(alpha_t);
    double eps_scale = (1.0 - alpha_t) / sqrt(1.0 - alpha_bar_t);
    *a = inv_sqrt_alpha;
    *b = -inv_sqrt_alpha * eps_scale;
    *c = sqrt(1.0 - alpha_t);
    return ORACLE_OK;
}

/* DDIM (Song, Meng, Ermon, ICLR 2021): the paper's C2I/T2I sampler (Sec. 4.1) is not
 * printed in it, so this follows the DDIM paper's generative step from alpha_bar_t to
 * alpha_bar_prev:
 *     x0_pred = (x_t - sqrt(1 - alpha_bar_t) eps) / sqrt(alpha_bar_t)
 *     x_prev  = sqrt(alpha_bar_prev) x0_pred + sqrt(1 - alpha_bar_prev - sigma^2) eps
 *               + sigma z
 *     sigma   = eta sqrt((1 - alpha_bar_prev) / (1 - alpha_bar_t))
 *                   sqrt(1 - alpha_bar_t / alpha_bar_prev)
 * collected as x_prev = a x_t + b eps + c z. */
int oracle_ddim_coefficients(double alpha_bar_t, double alpha_bar_prev, double eta, double *a,
                             double *b, double *c)
{
    if (!(alpha_bar_t > 0.0 && alpha_bar_t < 1.0) ||
        !(alpha_bar_prev >= alpha_bar_t && alpha_bar_prev <= 1.0) || !(eta >= 0.0))
        return ORACLE_BAD_ARG;
    double sigma = eta * sqrt((1.0 - alpha_bar_prev) / (1.0 - alpha_bar_t)) *
                   sqrt(1.0 - alpha_bar_t / alpha_bar_prev);
    double dir_var = 1.0 - alpha_bar_prev - sigma * sigma;
    if (dir_var < 0.0) return ORACLE_BAD_ARG;
    /* x0_pred contributes sqrt(abp)/sqrt(abt) * x_t and -sqrt(abp) sqrt(1-abt)/sqrt(abt) * eps */
    double x0_from_x = 1.0 / sqrt(alpha_bar_t);
    double x0_from_eps = -sqrt(1.0 - alpha_bar_t) / sqrt(alpha_bar_t);
    *a = sqrt(alpha_bar_prev) * x0_from_x;
    *b = sqrt(alpha_bar_prev) * x0_from_eps + sqrt(dir_var);
    *c = sigma;
    return ORACLE_OK;
}

/* Forecast of the cached model output followed by x <- a x + b v_hat + c z.  z may be NULL
 * (no noise term); x and z are stored in x_dtype.  bound[e] = |a x| + |b| sum_j |W_j||V_j|
 * + |c z|. */
void oracle_update(int v_dtype, const void *const *V, int m, const double *W, int64_t n,
                   double a, double b, double c, int x_dtype, const void *x, const void *z,
                   double *x_out, double *bound)
{
    for (int64_t e = 0; e < n; ++e) {
        double acc = 0.0, mag = 0.0;
        for (int j = 0; j < m; ++j) {
            double v = load_elem(v_dtype, V[j], e);
            acc += W[j] * v;
            mag += fabs(W[j]) * fabs(v);
        }
        double x0 = load_elem(x_dtype, x, e);
        double z0 = z ? load_elem(x_dtype, z, e) : 0.0;
        x_out[e] = a * x0 + b * acc + c * z0;
        if (bound) bound[e] = fabs(a * x0) + fabs(b) * mag + fabs(c * z0);
    }
}

/* ---------------------------------------------------------------------------------
 * Feature-probe drift of the adaptive schedule (Sec. 4.5): the relative L1 change
 *     out[0] = sum |cur - prev|,  out[1] = sum |prev|,  out[2] = out[0] / out[1]
 * (0 when both sums vanish, +inf when only the denominator does).
 * ------------------------------------------------------------------------------- */
void oracle_drift(int dtype, const void *cur, const void *prev, int64_t n, double *out)
{
    double num = 0.0, den = 0.0;
    for (int64_t e = 0; e < n; ++e) {
        double c = load_elem(dtype, cur, e), p = load_elem(dtype, prev, e);
        num += fabs(c - p);
        den += fabs(p);
    }
    out[0] = num;
    out[1] = den;
    /* Relative change; a probe with no magnitude has ratio 0 (no change) or +inf (any
     * change); a NaN anywhere in either tensor makes the ratio NaN. */
    if (den > 0.0)
        out[2] = num / den;
    else if (den == 0.0 && num == 0.0)
        out[2] = 0.0;
    else if (den == 0.0 && num > 0.0)
        out[2] = INFINITY;
    else
        out[2] = NAN;
}
