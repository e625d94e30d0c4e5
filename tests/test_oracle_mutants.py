"""Planted mistakes: each mutant of the oracle source must fail at least one pin.

A mutant is a copy of ``oracle/quasar_oracle.c`` with one plausible slip
(a dropped term, a wrong sign, a wrong rounding or tie rule, a transposed
operand), compiled on the CPU into a temporary directory and swapped in for
the real library while the pins of ``test_oracle_pins`` run against it.
"""
import ctypes
import os
import subprocess

import pytest

import oracle as oracle_mod
from tests import test_oracle_checker_pins as cpins
from tests import test_oracle_pins as pins

SRC = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))),
                   "oracle", "quasar_oracle.c")

MUTANTS = {
    "round half up": ("double k = nearbyint(t); /* default rounding mode: half to even */",
                      "double k = floor(t + 0.5);"),
    "symmetric round half up": ("double k = nearbyint(t);\n        if (k < -(double)Q)",
                                "double k = floor(t + 0.5);\n        if (k < -(double)Q)"),
    "offset sign": ("z = wbar - s * qbar;", "z = wbar + s * qbar;"),
    "error sign": ("const double d = s * (double)q[i] + z - (double)w[i];",
                   "const double d = s * (double)q[i] - z - (double)w[i];"),
    "unweighted denominator": ("den += hd[i] * dq * dq;", "den += dq * dq;"),
    "argmin ties to last": (
        "if (ek[k] < ek[best]) best = k;\n            double second = HUGE_VAL;\n"
        "            for (int k = 0; k < K; ++k) {\n                if (k == best) continue;\n"
        "                if (memcmp(qk + (size_t)k * G",
        "if (ek[k] <= ek[best]) best = k;\n            double second = HUGE_VAL;\n"
        "            for (int k = 0; k < K; ++k) {\n                if (k == best) continue;\n"
        "                if (memcmp(qk + (size_t)k * G"),
    "LUT argmin ties to last": (
        "if (ek[k] < ek[best]) best = k;\n            double second = HUGE_VAL;\n"
        "            for (int k = 0; k < K; ++k) {\n                if (k == best) continue;\n"
        "                if (memcmp(qk + (size_t)k * n",
        "if (ek[k] <= ek[best]) best = k;\n            double second = HUGE_VAL;\n"
        "            for (int k = 0; k < K; ++k) {\n                if (k == best) continue;\n"
        "                if (memcmp(qk + (size_t)k * n"),
    "NVFP4 argmin picks the largest error": (
        "if (ek[k] < ek[best]) best = k;\n            double second = HUGE_VAL;\n"
        "            for (int k = 0; k < K; ++k) {\n                if (k == best) continue;\n"
        "                if (sk[k]",
        "if (ek[k] > ek[best]) best = k;\n            double second = HUGE_VAL;\n"
        "            for (int k = 0; k < K; ++k) {\n                if (k == best) continue;\n"
        "                if (sk[k]"),
    "center sign": ("const double c = 0.5 * (mn + mx);", "const double c = 0.5 * (mx - mn);"),
    "clip ignored in offset": ("const double z = c - f * rho;", "const double z = c - rho;"),
    "EMA drops square": ("c1 * gi * gi", "c1 * gi"),
    "E4M3 subnormal exponent": ("ldexp((double)m / 8.0, -6)", "ldexp((double)m / 8.0, -7)"),
    "NVFP4 search scale": ("(double)clip[k] * amax_b / 6.0", "(double)clip[k] * amax_b / 4.0"),
    "NVFP4 error at unrounded scale": (
        "const double alpha = sT * e4m3_tab[sk[k]];",
        "const double alpha = (s2 == 0.0) ? sigma : s3 / s2;"),
    "degenerate step dropped": ("s = step;", "s = 0.0;"),
    "code margin not normalised": ("margin[i] = fabs(t - (j + 0.5)) / (double)qmax;",
                                   "margin[i] = fabs(t - (j + 0.5));"),
    "E2M1 ties to odd": ("if (d < bd || (d == bd && (m % 2) == 0)) {",
                         "if (d < bd || (d == bd && (m % 2) == 1)) {"),
    "AdamW without bias correction": ("lr * ((double)mi / bc1) / denom", "lr * (double)mi / denom"),
    "AdamW coupled weight decay": ("(double)w[i] * (1.0 - lr * wd) - lr", "(double)w[i] - lr * wd - lr"),
    "AdamW eps inside the root": ("sqrt((double)vi / bc2) + eps", "sqrt((double)vi / bc2 + eps)"),
    "symmetric argmin ties to last": ("best = (ek[k] < ek[best]) ? k : best;",
                                      "best = (ek[k] <= ek[best]) ? k : best;"),
    "symmetric fit with an offset": ("const double s = (s2 > 0.0) ? s3 / s2 : step;",
                                     "const double s = (s2 > 0.0) ? (s3 + 1e-3 * s2) / s2 : step;"),
    "symmetric grid on the full range": ("const double s = f * amax / (double)Q;",
                                         "const double s = 2.0 * f * amax / (double)(2 * Q + 1);"),
    "symmetric codes not clamped": ("if (k > (double)Q) k = (double)Q;\n        code[i]",
                                    "if (k > (double)(Q + 1)) k = (double)(Q + 1);\n        code[i]"),
    "LUT entry unweighted mean": ("W[q[i] & 7] += hd[i] * (double)w[i];", "W[q[i] & 7] += (double)w[i];"),
    "LUT entry sign dropped": ("return (x < 0.0 && mag != 0) ? (0x80 | mag) : mag;", "return mag;"),
    "LUT empty index at grid offset": ("lo + (double)k * s;", "lo + (double)(k + 1) * s;"),
    # mistakes in the single-candidate helpers the parity checker calls
    "refit D3 step over qmax + 1": ("const double step = (mx - mn) * (double)f / (double)qmax;",
                                    "const double step = (mx - mn) * (double)f / (double)(qmax + 1);"),
    "refit without the zero-saliency rule": (
        "group_saliency(h, G, hd);\n    const double step",
        "for (int i = 0; i < G; ++i) hd[i] = (double)h[i];\n    const double step"),
    "symmetric refit step over Q + 1": (
        "const double e = sym_fit(w, hd, code, G, Q, (double)f * amax / (double)Q, s_out);",
        "const double e = sym_fit(w, hd, code, G, Q, (double)f * amax / (double)(Q + 1), s_out);"),
    "NVFP4 helper codes keep a negative zero": ("const int neg = (w[i] < 0.0f) && m != 0;",
                                                "const int neg = (w[i] < 0.0f);"),
    "NVFP4 helper codes search scale": ("const double sigma = (double)f * amax_b / 6.0;",
                                        "const double sigma = (double)f * amax_b / 4.0;"),
    "NVFP4 helper scale fit unweighted": (
        "s3 += hd[i] * q * (double)w[i];\n    }\n    if (amax_b == 0.0)",
        "s3 += q * (double)w[i];\n    }\n    if (amax_b == 0.0)"),
    "NVFP4 helper N4 rule drops the factor": ("((double)f * amax_b / 6.0) / (double)s_T",
                                              "(amax_b / 6.0) / (double)s_T"),
    "NVFP4 helper error drops the tensor scale": (
        "const double alpha = (double)s_T * qo_e4m3_value(scale_bits);",
        "const double alpha = qo_e4m3_value(scale_bits);"),
    "LUT helper error reads the next entry": (
        "const double d = e4m3s_value(book[q[i] & 7]) - (double)w[i];",
        "const double d = e4m3s_value(book[(q[i] + 1) & 7]) - (double)w[i];"),
    "LUT helper fit grid origin": (
        "lut_entries(w, hd, n, c - (double)f * rho, 2.0 * (double)f * rho / 7.0, q, bk, book_margin);",
        "lut_entries(w, hd, n, c + (double)f * rho, 2.0 * (double)f * rho / 7.0, q, bk, book_margin);"),
    "LUT helper block ignores the factor": (
        "e = lut_candidate(w, hd, n, c, rho, (double)f, q, bk, margin, book_margin);",
        "e = lut_candidate(w, hd, n, c, rho, 1.0, q, bk, margin, book_margin);"),
    "LUT error at the grid point": ("const double d = e4m3s_value(book[q[i]]) - (double)w[i];\n        e += hd[i] * d * d;\n    }\n    return e;\n}\n\n/* Block range",
                                    "const double d = (lo + (double)q[i] * s) - (double)w[i];\n        e += hd[i] * d * d;\n    }\n    return e;\n}\n\n/* Block range"),
}

PIN_TESTS = [
    (pins.test_int_worked_examples, {}),
    (pins.test_nvfp4_worked_example, {}),
    (pins.test_codes_are_nearest_grid_level, {"bits": 3}),
    (pins.test_fit_matches_weighted_lstsq, {"bits": 3, "G": 128}),
    (pins.test_fit_normal_equations, {}),
    (pins.test_argmin_over_candidates, {}),
    (pins.test_single_salient_element_rule, {}),
    (pins.test_ema_special_cases, {}),
    (pins.test_e4m3_values_match_torch, {}),
    (pins.test_e2m1_grid_from_format, {}),
    (pins.test_nvfp4_fit_and_scale_are_optimal, {}),
    (pins.test_adamw_matches_torch_optimizer, {}),
    (pins.test_adamw_first_step_closed_form, {}),
    (pins.test_sym_worked_example, {}),
    (pins.test_sym_codes_are_nearest_levels_and_fit_is_lstsq, {"bits": 3}),
    (pins.test_sym_sign_symmetry_and_ties, {}),
    (pins.test_lut_worked_example, {}),
    (pins.test_lut_entries_are_the_best_e4m3_values, {}),
    (pins.test_lut_error_and_argmin, {}),
    (pins.test_lut_indices_follow_the_grid, {}),
    (cpins.test_refit_int_is_weighted_least_squares, {}),
    (cpins.test_refit_sym_is_least_squares_through_origin, {}),
    (cpins.test_codes_nvfp4_enumeration_and_kept_codes, {}),
    (cpins.test_fit_nvfp4_scale_enumerates_e4m3, {}),
    (cpins.test_eval_nvfp4_is_the_direct_error, {}),
    (cpins.test_lut_block_matches_app_b_candidates, {}),
    (cpins.test_lut_fit_is_the_weighted_mean_rounded, {}),
    (cpins.test_lut_eval_is_the_direct_error, {}),
]


def _build_mutant(tmp_path, old, new):
    src = open(SRC).read()
    assert src.count(old) == 1, f"mutation anchor not unique: {old!r}"
    path = tmp_path / "mutant.c"
    path.write_text(src.replace(old, new))
    so = tmp_path / "libmutant.so"
    subprocess.run(["gcc", "-O1", "-std=c11", "-fPIC", "-shared", "-ffp-contract=off",
                    str(path), "-o", str(so), "-lm"], check=True)
    return str(so)


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_pins_catch_planted_mistake(oracle, tmp_path, name):
    old, new = MUTANTS[name]
    so = _build_mutant(tmp_path, old, new)
    real = oracle_mod._load()
    lib = ctypes.CDLL(so)
    # give the mutant the same prototypes as the real library
    for sym in ("qo_ema", "qo_adamw", "qo_recon_int", "qo_refit_int", "qo_codes_int", "qo_tensor_scale",
                "qo_recon_nvfp4", "qo_e2m1_round", "qo_e4m3_round", "qo_e4m3_value",
                "qo_set_threads", "qo_get_threads", "qo_recon_lut", "qo_lut_block", "qo_lut_eval", "qo_lut_fit",
                "qo_recon_sym", "qo_codes_sym", "qo_refit_sym", "qo_codes_nvfp4",
                "qo_fit_nvfp4_scale", "qo_eval_nvfp4"):
        f_real, f_mut = getattr(real, sym), getattr(lib, sym)
        f_mut.argtypes, f_mut.restype = f_real.argtypes, f_real.restype
    caught = []
    oracle_mod._lib = lib
    try:
        for test, kw in PIN_TESTS:
            try:
                test(oracle_mod, **kw)
            except (AssertionError, ValueError, ZeroDivisionError, FloatingPointError):
                caught.append(test.__name__)
    finally:
        oracle_mod._lib = real
    assert caught, f"no pin caught the planted mistake '{name}'"
