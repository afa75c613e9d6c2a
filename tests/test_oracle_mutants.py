"""The pins catch plausible mistakes: each mutant of the oracle fails one.

A mutant is a copy of oracle.c with one planted mistake (a dropped term, a
wrong sign, a swapped operand, '>' for '>=', a reversed order or tie rule, a
wrong residual), compiled to a temporary library. The pin tests run against
it with the module's loaded library swapped; at least one must fail. CPU only.
"""
import contextlib
import ctypes
import os
import subprocess

import pytest

import oracle
import test_oracle_pins as pins

_SRC = os.path.join(os.path.dirname(oracle.__file__), "oracle.c")

MUTANTS = {
    "two_step_rounding": [("fmaf(gamma, gj, e[j])", "(gamma * gj + e[j])")],
    "swapped_operands": [("fmaf(gamma, gj, e[j])", "fmaf(gamma, e[j], gj)")],
    "dropped_error_term": [("fmaf(gamma, gj, e[j])", "fmaf(gamma, gj, 0.0f)")],
    "wrong_sign": [("fmaf(gamma, gj, e[j])", "fmaf(-gamma, gj, e[j])")],
    "strict_threshold": [("(fabsf(a) >= lambda)", "(fabsf(a) > lambda)")],
    "sends_zeros": [("&& (a != 0.0f)", "")],
    "residual_not_cleared": [("      e[j] = 0.0f;                                       /* R7 */",
                              "      e[j] = a;")],
    "topk_smallest_first": [("if (m != 0) return -m;", "if (m != 0) return m;")],
    "topk_highest_index_ties": [("  return (ia > ib) - (ia < ib);", "  return (ia < ib) - (ia > ib);")],
    "topk_residual_kept": [("    e[j] = 0.0f;                                      /* R7 */",
                            "    e[j] = a[j];")],
    "nan_ranked_by_payload": [("    if (nx && ny) return 0;",
                               "    if (nx && ny) { uint32_t px, py; memcpy(&px, &ax, 4);"
                               " memcpy(&py, &ay, 4); return (px > py) - (px < py); }")],
    "aggregate_reverse_order": [("for (uint32_t i = 0; i < n; ++i) {",
                                 "for (uint32_t i = n; i-- > 0;) {")],
    "nan_ranks_lowest": [("    return nx ? 1 : -1;", "    return nx ? -1 : 1;")],
    "layerwise_local_indices": [("idx[sent + p] += (uint32_t)lo;", "idx[sent + p] += 0u;")],
    "layerwise_first_k_everywhere": [("                       seg_k[s], hi - lo,",
                                      "                       seg_k[0] < hi - lo ? seg_k[0] : hi - lo, hi - lo,")],
    "layerwise_error_not_sliced": [("e + lo, gamma,", "e, gamma,")],
    "update_uses_old_momentum": [
        ("        m[j] = fmaf(mu, m[j], delta);                /* m <- mu m + Delta' */\n"
         "        float u = delta + m[j];                      /* Delta' + m */",
         "        float u = delta + m[j];                      /* Delta' + m */\n"
         "        m[j] = fmaf(mu, m[j], delta);                /* m <- mu m + Delta' */")],
    "update_alpha_dropped": [("float delta = alpha * s[j];", "float delta = s[j];")],
    "update_momentum_two_step": [("fmaf(mu, m[j], delta)", "(mu * m[j] + delta)")],
    "update_wrong_sign": [("fmaf(-lr, u, x[j])", "fmaf(lr, u, x[j])")],
    "update_sgd_adds": [("x[j] = x[j] - delta;", "x[j] = x[j] + delta;")],
    "round_half_away": [("float r = rintf(s);", "float r = roundf(s);")],
    "round_truncate": [("float r = rintf(s);", "float r = truncf(s);")],
    "round_residual_not_subtracted": [("e[j] = a - c;", "e[j] = a;")],
    # the bf16 widening inside the scaled-rounding step only (the line is
    # followed there by the scaling, not by the threshold or the sort)
    "round_bf16_integer_value": [
        ("bf16_bits_to_float(g_bf16[j]);\n    float a = fmaf(gamma, gj, e[j]);"
         "                           /* R2 */\n    float s = ldexpf(a, m);",
         "(float)g_bf16[j];\n    float a = fmaf(gamma, gj, e[j]);"
         "                           /* R2 */\n    float s = ldexpf(a, m);")],
    "round_bf16_sign_dropped": [
        ("bf16_bits_to_float(g_bf16[j]);\n    float a = fmaf(gamma, gj, e[j]);"
         "                           /* R2 */\n    float s = ldexpf(a, m);",
         "bf16_bits_to_float(g_bf16[j] & 0x7fff);\n    float a = fmaf(gamma, gj, e[j]);"
         "                           /* R2 */\n    float s = ldexpf(a, m);")],
    "bf16_widening_shift": [("((uint32_t)bits) << 16", "((uint32_t)bits) << 15")],
    "round_scale_sign": [("float s = ldexpf(a, m);", "float s = ldexpf(a, -m);")],
    "round_saturates_instead": [("      q[j] = 0;                                                /* not representable: */",
                                 "      q[j] = a > 0 ? 2147483647 : -2147483647;")],
    "int_aggregate_in_float": [("    int64_t s = 0;\n    for (uint32_t i = 0; i < n; ++i) s += q[i][j];",
                                "    float s = 0;\n    for (uint32_t i = 0; i < n; ++i) s += (float)q[i][j];")],
    "error_norm_fp32_square": [("s += (double)e[j] * (double)e[j];", "s += (double)(e[j] * e[j]);")],
    "error_norm_abs": [("s += (double)e[j] * (double)e[j];", "s += fabs((double)e[j]);")],
}

PIN_TESTS = [
    pins.test_accumulate_is_one_rounded_fma,
    pins.test_accumulate_operand_roles,
    pins.test_ht_threshold_is_inclusive,
    pins.test_ht_lambda_zero_sends_exactly_the_nonzeros,
    pins.test_ht_nan_and_inf,
    lambda: pins.test_ht_reconstruction_and_absolute_bound(3001),
    lambda: pins.test_topk_matches_bruteforce_optimum(0),
    lambda: pins.test_topk_matches_bruteforce_optimum(1),
    pins.test_topk_matches_stable_argsort_with_ties,
    pins.test_topk_special_cases,
    pins.test_topk_nan_inf_order,
    pins.test_aggregate_sums_in_worker_order,
    lambda: pins.test_error_feedback_conserves_mass("ht"),
    pins.test_topk_layerwise_hand_example,
    lambda: pins.test_topk_layerwise_matches_bruteforce_per_segment(0),
    lambda: pins.test_topk_layerwise_matches_bruteforce_per_segment(1),
    pins.test_update_algorithm1_subtracts_the_mean,
    pins.test_update_momentum_closed_form,
    pins.test_update_momentum_zero_factor,
    pins.test_update_rounding_follows_r12,
    pins.test_error_norm_hand_values_and_exactness,
    pins.test_error_norm_bounds_of_the_sparsifiers,
    pins.test_scaled_round_hand_example,
    pins.test_scaled_round_is_an_absolute_compressor,
    pins.test_scaled_round_unsent_coordinates,
    pins.test_scaled_round_bf16_hand_example,
    pins.test_scaled_round_bf16_is_the_widened_fp32,
    pins.test_ht_bf16_widening,
    pins.test_int_aggregate_is_exact_and_order_free,
]


@contextlib.contextmanager
def _swapped_library(path):
    oracle._load()
    saved = oracle._lib
    lib = ctypes.CDLL(path)
    # reuse the argtypes of the real library
    for name in ("oracle_ef_hard_threshold", "oracle_ef_hard_threshold_bf16",
                 "oracle_ef_topk", "oracle_ef_topk_bf16", "oracle_ef_topk_layerwise",
                 "oracle_ef_topk_layerwise_bf16", "oracle_sparse_aggregate",
                 "oracle_sparse_aggregate_apply", "oracle_error_norm_sq",
                 "oracle_ef_scaled_round", "oracle_ef_scaled_round_bf16",
                 "oracle_int_aggregate"):
        fn, ref = getattr(lib, name), getattr(saved, name)
        fn.argtypes, fn.restype = ref.argtypes, ref.restype
    oracle._lib = lib
    try:
        yield
    finally:
        oracle._lib = saved


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_mutant_is_caught(name, tmp_path):
    src = open(_SRC).read()
    for old, new in MUTANTS[name]:
        assert old in src, (name, old)
        src = src.replace(old, new)
    c_path = tmp_path / "mutant.c"
    c_path.write_text(src)
    so_path = str(tmp_path / "libmutant.so")
    subprocess.run(["gcc", *oracle._CFLAGS, "-o", so_path, str(c_path), "-lm"], check=True)
    failures = 0
    with _swapped_library(so_path):
        for t in PIN_TESTS:
            try:
                t()
            except AssertionError:
                failures += 1
    assert failures >= 1, "mutant %s survived every pin" % name
