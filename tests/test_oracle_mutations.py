"""The oracle's pins catch plausible mistakes.

Each case plants one mistake (a dropped term, a wrong index, a wrong sign, an
off-by-one in an exponent or a period test, ...) in a temporary copy of the
oracle's C source, rebuilds that copy, and runs the pin suite against it in
a subprocess.  The suite must fail for every planted mistake.  Nothing here
touches the real oracle or any GPU.
"""
import os
import shutil
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
SRC = os.path.join(ROOT, "oracle", "mtdao_oracle.c")

MUTATIONS = {
    "bias_correction_exponent_t": ("pow(b, (double)(t + 1))", "pow(b, (double)(t))"),
    "eps_inside_sqrt": ("(sqrt(v_new / corr_v) + c->eps)", "sqrt(v_new / corr_v + c->eps)"),
    "second_moment_of_clipped_grad": (
        "(1.0 - c->beta2) * g * g;\n    v[k] = v_new;\n    double corr_v",
        "(1.0 - c->beta2) * g_hat * g_hat;\n    v[k] = v_new;\n    double corr_v"),
    "omega_paired_with_wrong_momentum": ("combo += c->omega[j] * (u_new / corr);",
                                         "combo += c->omega[c->n_mom - 1 - j] * (u_new / corr);"),
    "gradient_term_dropped": ("double combo = (1.0 - sum_omega) * g_hat;", "double combo = 0.0;"),
    "adam_update_sign": ("x[k] = x[k] - lr * delta;\n    return x[k];\n}\n\n/* Algorithm 2",
                         "x[k] = x[k] + lr * delta;\n    return x[k];\n}\n\n/* Algorithm 2"),
    "adopt_normalises_with_old_v": ("g_hat = g / (sqrt(v_new) + c->eps);",
                                    "g_hat = g / (sqrt(c->beta2 * v_new) + c->eps);"),
    "adopt_original_order_uses_new_v": (
        "        g_hat = g / (sqrt(v[k]) + c->eps);\n        v[k] = c->beta2 * v[k] + (1.0 - c->beta2) * g * g;",
        "        v[k] = c->beta2 * v[k] + (1.0 - c->beta2) * g * g;\n        g_hat = g / (sqrt(v[k]) + c->eps);"),
    "adopt_original_order_clamp_index": ("update_index = t - 1;", "update_index = t;"),
    "adopt_clamp_missing": ("if (g_tilde > ct) g_tilde = ct;", "if (0) g_tilde = ct;"),
    "mean_divides_by_M_minus_1": (
        "double mean = sum / (double)M;\n        for (int m = 0; m < M; ++m)\n            s[",
        "double mean = sum / (double)(M > 1 ? M - 1 : 1);\n        for (int m = 0; m < M; ++m)\n            s["),
    "sync_phase_off_by_one": (
        "    if (divides(c->period_x, t)) mask |= bit_x();\n    for (int j = 0; j < c->n_mom; ++j)\n"
        "        if (divides(c->period_u[j], t)) mask |= bit_u(j);",
        "    if (divides(c->period_x, t + 1)) mask |= bit_x();\n    for (int j = 0; j < c->n_mom; ++j)\n"
        "        if (divides(c->period_u[j], t + 1)) mask |= bit_u(j);"),
    "clip_constant": ("double f = c->clip_rho / (norm + 1e-6);", "double f = c->clip_rho / (norm + 1e-3);"),
    "adopt_beta_index": ("double u_new = b * u_j[j][k] + (1.0 - b) * g_tilde;",
                         "double u_new = c->beta1[0] * u_j[j][k] + (1.0 - c->beta1[0]) * g_tilde;"),
    "sgdm_momentum_scaled": (
        "        double u_new = b * u_j[j][k] + (1.0 - b) * g_hat;\n        u_j[j][k] = u_new;\n"
        "        delta += c->omega[j] * u_new;\n    }\n    x[k] = x[k] - lr * delta;\n    return x[k];\n}\n\n/*\n * One",
        "        double u_new = b * u_j[j][k] + (1.0 - b) * g_hat * 0.999;\n        u_j[j][k] = u_new;\n"
        "        delta += c->omega[j] * u_new;\n    }\n    x[k] = x[k] - lr * delta;\n    return x[k];\n}\n\n/*\n * One"),
    "v_sync_skipped": ("    if (c->base != MTO_SGDM && (mask & bit_v(c)))\n        mto_mean_over_workers(M, n, v);",
                       "    if (0)\n        mto_mean_over_workers(M, n, v);"),
    "variance_over_M_minus_1": ("out[0] += (v - mean) * (v - mean) / (double)M;",
                                "out[0] += (v - mean) * (v - mean) / (double)(M - 1);"),
    "dot_with_worker_instead_of_mean": ("out[2 + M + m] += v * mean;", "out[2 + M + m] += v * v;"),
    "half_life_period_truncated": ("long long k = (long long)floor(mto_half_life(beta) + 0.5);",
                                   "long long k = (long long)floor(mto_half_life(beta));"),
    "half_life_period_not_floored_at_kx": ("return k < period_x ? period_x : k;", "return k;"),
    "comm_reduction_without_v": ("if (c->base != MTO_SGDM && c->period_v > 0) per_step",
                                 "if (0 && c->period_v > 0) per_step"),
    "global_pseudo_grad_without_anchor": ("double global = sum / (double)M - a[i];",
                                          "double global = sum / (double)M;"),
}


@pytest.mark.parametrize("name", sorted(MUTATIONS))
def test_pins_catch_planted_mistake(name, tmp_path):
    src = open(SRC).read()
    old, new = MUTATIONS[name]
    assert src.count(old) == 1, "mutation site not found: %s" % name
    work = tmp_path / "repo"
    for sub in ("oracle", "synth", "tests"):
        shutil.copytree(os.path.join(ROOT, sub), work / sub,
                        ignore=shutil.ignore_patterns("_build", "__pycache__"))
    (work / "oracle" / "mtdao_oracle.c").write_text(src.replace(old, new))
    r = subprocess.run([sys.executable, "-m", "pytest", "-q", "-x", "-p", "no:cacheprovider",
                        "tests/test_oracle_pins.py"], cwd=work, capture_output=True, text=True,
                       timeout=600)
    assert r.returncode != 0, "planted mistake %s passed every pin:\n%s" % (name, r.stdout[-2000:])
    assert "failed" in r.stdout
