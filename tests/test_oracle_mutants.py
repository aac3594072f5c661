"""The oracle's pins catch plausible mistakes.

Each case plants one slip in a copy of oracle/oracle.c (a dropped term, a wrong index or sign,
a transposed operand, the printed-but-contradicted reading of Eq. 12 ...), compiles it on the CPU
and runs the pin suites against that build; at least one pin must fail.  The real oracle is
never modified.
"""
import os
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
SRC = os.path.join(ROOT, "oracle", "oracle.c")
PINS = ["tests/test_oracle_pins.py", "tests/test_oracle_samplers.py"]

MUTANTS = {
    # Eq. 8: trapezoid factor only at the newest end
    "eq8_end_factor": ("cfac[j - 1] = (j == 1 || j == m) ? 0.5 : 1.0;",
                       "cfac[j - 1] = (j == 1) ? 0.5 : 1.0;"),
    # Eq. 9: node times paired with the wrong nodes (reversed order)
    "eq9_wrong_node": ("u[j - 1] = cfac[j - 1] * sign / (t - s[j - 1]);",
                       "u[j - 1] = cfac[j - 1] * sign / (t - s[m - j]);"),
    # Eq. 9: no alternating sign
    "eq9_no_alternation": ("double sign = (j % 2 == 0) ? 1.0 : -1.0;", "double sign = 1.0;"),
    # Eq. 10: clip left out
    "eq10_no_clip": ("ut[j] = fmax(-C, fmin(C, u[j]));", "ut[j] = u[j];"),
    # Eq. 11: sign of u~ dropped
    "eq11_no_sign": ("a[j] = sgn_plus(ut[j]) * pow(fabs(ut[j]) + eta, delta);",
                     "a[j] = pow(fabs(ut[j]) + eta, delta);"),
    # Eq. 11: power on the wrong quantity (eta outside, delta ignored)
    "eq11_power_ignored": ("a[j] = sgn_plus(ut[j]) * pow(fabs(ut[j]) + eta, delta);",
                           "a[j] = sgn_plus(ut[j]) * (fabs(ut[j]) + eta);"),
    # Eqs. 10-11 in the wrong order: the power applied first and its result clipped
    "eq10_after_eq11": ("    for (int j = 0; j < m; ++j) ut[j] = fmax(-C, fmin(C, u[j]));\n\n"
                        "    /* Eq. 11 */\n    double sum = 0.0, sum_abs = 0.0;\n"
                        "    for (int j = 0; j < m; ++j) {\n"
                        "        a[j] = sgn_plus(ut[j]) * pow(fabs(ut[j]) + eta, delta);",
                        "    for (int j = 0; j < m; ++j) ut[j] = u[j];\n\n"
                        "    /* Eq. 11 */\n    double sum = 0.0, sum_abs = 0.0;\n"
                        "    for (int j = 0; j < m; ++j) {\n"
                        "        a[j] = fmax(-C, fmin(C, sgn_plus(ut[j]) * pow(fabs(ut[j]) + eta, delta)));"),
    # Eq. 11: the decay power inverted
    "eq11_power_inverted": ("a[j] = sgn_plus(ut[j]) * pow(fabs(ut[j]) + eta, delta);",
                            "a[j] = sgn_plus(ut[j]) * pow(fabs(ut[j]) + eta, 1.0 / delta);"),
    # Eq. 12 as printed: the last weight scaled by lambda instead of a blend towards x_{f=-1}
    "eq12_printed_vector": ("W[j] = (1.0 - lambda) * alpha + (j == 0 ? lambda : 0.0);",
                            "W[j] = (j < m - 1 ? (1.0 - lambda) : lambda) * alpha;"),
    # Lagrange: wrong index in the numerator
    "lagrange_index": ("prod *= (t - s[k]) / (s[j] - s[k]);",
                       "prod *= (t - s[j]) / (s[j] - s[k]);"),
    # Eq. 13: weights paired with the nodes in reverse
    "eq13_transposed": ("            acc += W[j] * v;\n            mag += fabs(W[j]) * fabs(v);\n        }\n        out[e] = acc;",
                        "            acc += W[m - 1 - j] * v;\n            mag += fabs(W[j]) * fabs(v);\n        }\n        out[e] = acc;"),
    # Eq. 13: oldest node dropped
    "eq13_dropped_term": ("void oracle_combine(int dtype, const void *const *F, int m, const double *W, int64_t n,\n                    double *out, double *bound)\n{\n    for (int64_t e = 0; e < n; ++e) {\n        double acc = 0.0, mag = 0.0;\n        for (int j = 0; j < m; ++j) {",
                          "void oracle_combine(int dtype, const void *const *F, int m, const double *W, int64_t n,\n                    double *out, double *bound)\n{\n    for (int64_t e = 0; e < n; ++e) {\n        double acc = 0.0, mag = 0.0;\n        for (int j = 0; j < m - 1; ++j) {"),
    # Euler: wrong sign of the step
    "euler_sign": ("x_out[e] = x0 + dt * acc;", "x_out[e] = x0 - dt * acc;"),
    # bf16 widening: wrong shift
    "bf16_shift": ("uint32_t word = ((uint32_t)bits) << 16;", "uint32_t word = ((uint32_t)bits) << 15;"),
    # Eq. 3: alpha_t and alpha_bar_t transposed in the noise coefficient
    "ddpm_transposed": ("double eps_scale = (1.0 - alpha_t) / sqrt(1.0 - alpha_bar_t);",
                        "double eps_scale = (1.0 - alpha_bar_t) / sqrt(1.0 - alpha_t);"),
    # DDIM: wrong sign of the direction term
    "ddim_direction_sign": ("*b = sqrt(alpha_bar_prev) * x0_from_eps + sqrt(dir_var);",
                            "*b = sqrt(alpha_bar_prev) * x0_from_eps - sqrt(dir_var);"),
    # drift: difference of magnitudes instead of magnitude of the difference
    "drift_abs": ("num += fabs(c - p);", "num += fabs(c) - fabs(p);"),
    # update: noise term dropped
    "update_no_noise": ("x_out[e] = a * x0 + b * acc + c * z0;", "x_out[e] = a * x0 + b * acc;"),
}


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_pins_catch_the_mutant(name, tmp_path):
    old, new = MUTANTS[name]
    src = open(SRC).read()
    assert src.count(old) == 1, f"mutation site for {name} not found exactly once"
    mut = tmp_path / "oracle_mut.c"
    mut.write_text(src.replace(old, new))
    lib = tmp_path / "liboracle_mut.so"
    subprocess.check_call(["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-fno-fast-math",
                           "-ffp-contract=off", "-o", str(lib), str(mut), "-lm"])
    env = dict(os.environ, ORACLE_LIB=str(lib))
    p = subprocess.run([sys.executable, "-m", "pytest", "-x", "-q", "-p", "no:cacheprovider",
                        *PINS], cwd=ROOT, env=env, capture_output=True, text=True, timeout=600)
    assert p.returncode != 0, f"no pin failed for mutant {name}:\n{p.stdout[-2000:]}"
    assert "failed" in p.stdout
