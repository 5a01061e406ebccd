"""Planted mistakes in the oracle must be caught by the pins (CPU only).

Each case copies oracle/bla_oracle.c, plants one plausible mistake (a wrong sign,
a dropped term, an index or grid error, a transposed operand), compiles the copy
and runs every pin against it; at least one pin must fail.  This shows the pins
constrain every part of the oracle, not only the parts they were written for.
"""
import ctypes
import os
import subprocess
import sys

import pytest

sys.path.insert(0, os.path.dirname(os.path.abspath(__file__)))
import oracle_pins as P  # noqa: E402

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
SRC = os.path.join(ROOT, "oracle", "bla_oracle.c")

MUTANTS = {
    "rotation_sign": ("xc[i] = cw * a - sw * b + x[i];", "xc[i] = cw * a + sw * b + x[i];"),
    "input_into_sin_row": ("xc[i] = cw * a - sw * b + x[i];\n            xs[i] = sw * a + cw * b;",
                           "xc[i] = cw * a - sw * b;\n            xs[i] = sw * a + cw * b + x[i];"),
    "coefficient_factor": ("A[j * M + m] = 2.0 * cos", "A[j * M + m] = 1.0 * cos"),
    "sin_coefficient_sign": ("B[j * M + m] = 2.0 * sin", "B[j * M + m] = -2.0 * sin"),
    "mode0_coefficient": ("A[j * M + 0] = 1.0 / n;", "A[j * M + 0] = 2.0 / n;"),
    "mask_strict": ("(double)tabs >= delta[j]", "(double)tabs > delta[j]"),
    "grid_floor": ("nearbyint((double)j * Te / (double)S)", "floor((double)j * Te / (double)S)"),
    "no_period_clamp": ("return T < r ? r : T;", "return T;"),
    "scale_1_over_d": ("1.0 / sqrt((double)dk)", "1.0 / (double)dk"),
    "swapped_A_B_readout": ("acc += A[j * M + m] * Kc[m * dk + i] + B[j * M + m] * Ks[m * dk + i];",
                            "acc += B[j * M + m] * Kc[m * dk + i] + A[j * M + m] * Ks[m * dk + i];"),
    "read_before_update": ("rotate_add(M, dk, c->w, Kc, Ks, k + (size_t)t * dk);\n        rotate_add(M, dv, c->w, Vc, Vs, v + (size_t)t * dv);\n        if (want && !want[t]) continue;\n        /* \"Compute",
                           "rotate_add(M, dk, c->w, Kc, Ks, k + (size_t)(t > 0 ? t - 1 : 0) * dk);\n        rotate_add(M, dv, c->w, Vc, Vs, v + (size_t)t * dv);\n        if (want && !want[t]) continue;\n        /* \"Compute"),
    "backward_no_scale": ("dP *= c->scale;", "dP *= 1.0;"),
    "backward_no_centering": ("p[j] * (dp[j] - pdp) * wgt", "p[j] * dp[j] * wgt"),
    "dirichlet_no_factor2": ("acc += 2.0 / n * cos(m * w * x);", "acc += 1.0 / n * cos(m * w * x);"),
    "absolute_interp_sign": ("+ sin(t * m * c->w) * B[j * M + m];", "- sin(t * m * c->w) * B[j * M + m];"),
    "absolute_backward_lag_weight": ("return absolute ? u - dj : t - u - dj;", "return t - u - dj;"),
    "decay_after_add": ("Kp[j * dk + e] = keep * Kp[j * dk + e] + ip[j] * k[(size_t)i * dk + e];",
                        "Kp[j * dk + e] = keep * (Kp[j * dk + e] + ip[j] * k[(size_t)i * dk + e]);"),
    "decay_relative_phase": ("double t = (double)(c->pos0 + i);", "double t = (double)i;"),
    "decay_factor_sign": ("double keep = 1.0 - ip[j];", "double keep = 1.0 + ip[j];"),
    "decay_backward_product_inclusive": ("Wt[(size_t)u * S + j] = ip[(size_t)u * S + j] * prod;\n                prod *= 1.0 - ip[(size_t)u * S + j];",
                                         "prod *= 1.0 - ip[(size_t)u * S + j];\n                Wt[(size_t)u * S + j] = ip[(size_t)u * S + j] * prod;"),
    "selection_skips_state": ("rotate_add(M, dk, c->w, Kc, Ks, k + (size_t)t * dk);\n        rotate_add(M, dv, c->w, Vc, Vs, v + (size_t)t * dv);\n        if (want && !want[t]) continue;\n        const double *qt",
                              "if (want && !want[t]) continue;\n        rotate_add(M, dk, c->w, Kc, Ks, k + (size_t)t * dk);\n        rotate_add(M, dv, c->w, Vc, Vs, v + (size_t)t * dv);\n        const double *qt"),
    "explicit_omega_ignored": ("return omega > 0.0 ? omega : 2.0 * ORC_PI / orc_period(M, T);",
                               "return 2.0 * ORC_PI / orc_period(M, T);"),
    "explicit_scale_ignored": ("c.scale = scale > 0.0 ? scale : 1.0 / sqrt((double)dk);",
                               "c.scale = 1.0 / sqrt((double)dk);"),
    "decay_value_not_decayed": ("Vp[j * dv + e] = keep * Vp[j * dv + e] + ip[j]", "Vp[j * dv + e] = Vp[j * dv + e] + ip[j]"),
    # state layout on the way in and out, the mode read-out, the log-sum-exp
    "store_state_swapped_rows": ("memcpy(sk + (size_t)(2 * m) * dk, Kc + m * dk, sizeof(double) * dk);\n        memcpy(sk + (size_t)(2 * m + 1) * dk, Ks + m * dk, sizeof(double) * dk);",
                                 "memcpy(sk + (size_t)(2 * m) * dk, Ks + m * dk, sizeof(double) * dk);\n        memcpy(sk + (size_t)(2 * m + 1) * dk, Kc + m * dk, sizeof(double) * dk);"),
    "load_state_value_rows_swapped": ("memcpy(Vc + m * dv, sv + (size_t)(2 * m) * dv, sizeof(double) * dv);\n        memcpy(Vs + m * dv, sv + (size_t)(2 * m + 1) * dv, sizeof(double) * dv);",
                                      "memcpy(Vc + m * dv, sv + (size_t)(2 * m + 1) * dv, sizeof(double) * dv);\n        memcpy(Vs + m * dv, sv + (size_t)(2 * m) * dv, sizeof(double) * dv);"),
    "modes_readout_swapped": ("acc += uc[m] * Vc[m * dv + i] + us[m] * Vs[m * dv + i];", "acc += uc[m] * Vs[m * dv + i] + us[m] * Vc[m * dv + i];"),
    "lse_without_max": ("return mx + log(sum);", "return log(sum);"),
    "lse_base2": ("return mx + log(sum);", "return mx + log2(sum);"),
    # the VJPs: a transposed operand, a dropped weight, an off-by-one causal range, a dropped centering
    "backward_dk_transposed_operand": ("dk_[(size_t)u * dk + i] += dP * qt[i];\n            }\n            for (int i = 0; i < dv; ++i) dv_[(size_t)u * dv + i] += g * dot[i];\n        }\n    }\n    free(Dt);",
                                       "dk_[(size_t)u * dk + i] += dP * k[(size_t)u * dk + i];\n            }\n            for (int i = 0; i < dv; ++i) dv_[(size_t)u * dv + i] += g * dot[i];\n        }\n    }\n    free(Dt);"),
    "backward_dv_unweighted": ("double wgt = Dt[weight_arg(absolute, t, u, (int)delta[j]) + off];\n                g += p[j] * wgt;",
                               "double wgt = Dt[weight_arg(absolute, t, u, (int)delta[j]) + off];\n                g += p[j];"),
    "backward_excludes_current_token": ("for (int u = 0; u <= t; ++u) {\n            double g = 0.0, dP = 0.0;\n            for (int j = 0; j < S; ++j) {\n                double wgt = Dt[",
                                        "for (int u = 0; u < t; ++u) {\n            double g = 0.0, dP = 0.0;\n            for (int j = 0; j < S; ++j) {\n                double wgt = Dt["),
    "decay_backward_no_centering": ("double wgt = Wt[(size_t)u * S + j];\n                g += p[j] * wgt;\n                dP += p[j] * (dp[j] - pdp) * wgt;",
                                    "double wgt = Wt[(size_t)u * S + j];\n                g += p[j] * wgt;\n                dP += p[j] * dp[j] * wgt;"),
}


@pytest.fixture(scope="module")
def src_text():
    with open(SRC) as f:
        return f.read()


@pytest.mark.filterwarnings("ignore::RuntimeWarning")   # a broken oracle may yield NaN; the pins count it as a failure
@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_mutant_is_caught(name, src_text, tmp_path, monkeypatch):
    import oracle.oracle as oo
    old, new = MUTANTS[name]
    assert src_text.count(old) >= 1, "mutation anchor not found: " + name
    (tmp_path / "m.c").write_text(src_text.replace(old, new))
    lib_path = str(tmp_path / "libm.so")
    subprocess.run(["gcc", "-O1", "-fPIC", "-shared", "-fopenmp", "-std=c11", "-o", lib_path,
                    str(tmp_path / "m.c"), "-lm"], check=True)
    monkeypatch.setattr(oo, "_lib", oo._configure(ctypes.CDLL(lib_path)))
    failed = []
    for pname, (fn, tol) in sorted(P.ALL_PINS.items()):
        try:
            err = fn(oo)
        except Exception:            # a crash or rejected argument also counts as caught
            err = float("inf")
        if not err <= tol:
            failed.append(pname)
    assert failed, "planted mistake %r passed every pin" % name


def test_per_head_period_mapping_mutant_is_caught(monkeypatch):
    """A front end that hands each head another head's period (reversed order) fails the
    per-head pins."""
    import oracle
    import oracle.oracle as oo
    real = oo._by_head

    def swapped(fn, Ts, arrays, H, **kw):
        return real(fn, Ts[::-1].copy(), arrays, H, **kw)

    monkeypatch.setattr(oo, "_by_head", swapped)
    assert P.pin_per_head_period(oracle) > 1e-3
