"""The oracle's pins are strong enough: plant a plausible mistake in a copy of the
oracle (a dropped term, a wrong sign or index, a flipped tie rule, an unweighted
mean, ...), rebuild it, and check that at least one pin of tests/test_oracle.py
fails. The unmodified copy must pass every pin, which validates the harness."""
import ctypes
import os

import pytest

import oracle
import test_oracle as pins

SRC = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "oracle", "kq_oracle.c")

MUTANTS = {
    "assign_tie_to_highest": ("if (d < best) {\n                best = d;\n                bk = k;",
                              "if (d <= best) {\n                best = d;\n                bk = k;"),
    "distance_drops_last_term": ("    for (int j = 0; j < KQO_D; ++j) {\n        float t = x[j] - c[j];",
                                 "    for (int j = 0; j < KQO_D - 1; ++j) {\n        float t = x[j] - c[j];"),
    "distance_sign_error": ("float t = x[j] - c[j];", "float t = x[j] + c[j];"),
    "mean_divides_by_z_plus_1": ("z[k] > 0 ? (float)(sum[e] / (double)z[k])", "z[k] > 0 ? (float)(sum[e] / (double)(z[k] + 1))"),
    "empty_cluster_zeroed": (": C_prev[e];", ": 0.0f;"),
    "update_wrong_coordinate": ("+= (double)W[i * KQO_D + j];", "+= (double)W[i * KQO_D + (j + 1) % KQO_D];"),
    "levels_ignore_weights": ("wsum[cur[m]] += z;\n            qsum[cur[m]] += z * q[m];",
                              "wsum[cur[m]] += 1;\n            qsum[cur[m]] += q[m];"),
    "level_init_off_by_one": ("(double)l / 63.0", "(double)l / 64.0"),
    "level_tie_to_higher": ("if (d < best) {\n            best = d;\n            bl = l;",
                            "if (d <= best) {\n            best = d;\n            bl = l;"),
    "level_fit_never_converges": ("if (it > 0 && memcmp(cur, prev, (size_t)N) == 0) break;", "if (0) break;"),
    "reconstruct_reversed_row": ("C[k * KQO_D + j];", "C[k * KQO_D + (KQO_D - 1 - j)];"),
    "objective_squares": ("J += (double)dist[i];", "J += (double)dist[i] * (double)dist[i];"),
    "grad_step_sign_error": ("C_next[e] = C[e] - step;", "C_next[e] = C[e] + step;"),
    "grad_step_divides_by_z_plus_1": ("float mean = (float)(sum[e] / (double)z[k]);",
                                      "float mean = (float)(sum[e] / (double)(z[k] + 1));"),
    "grad_step_empty_zeroed": ("C_next[e] = C[e];\n            }", "C_next[e] = 0.0f;\n            }"),
    "grad_step_skips_lr": ("float step = lr * mean;\n                C_next", "float step = mean;\n                C_next"),
    "levels_grad_wrong_coordinate": ("int l = codes[(int64_t)k * KQO_D + j];",
                                     "int l = codes[(int64_t)k * KQO_D + (j + 1) % KQO_D];"),
    "levels_grad_sign_error": ("levels_next[l] = levels[l] - step;", "levels_next[l] = levels[l] + step;"),
    "levels_grad_counts_kernels": ("z[l] += 1;\n            sum[l]", "z[l] += (j == 0);\n            sum[l]"),
    "scalar_fit_zero_weight": ("return w ? (int64_t)w[m / group] : 1;", "return w ? (int64_t)w[m / group] : 0;"),
}

PINS = [
    lambda: pins.test_assign_brute_force_integers(64, 16, 0),
    lambda: pins.test_assign_brute_force_integers(37, 5, 1),
    pins.test_assign_constructed_ties,
    pins.test_assign_float_against_exact,
    pins.test_update_mean_of_members_exact,
    pins.test_update_dyadic_bit_exact,
    pins.test_k1_global_mean,
    pins.test_k_equals_n_identity,
    pins.test_fit_objective_non_increasing_and_consistent,
    pins.test_level_fit_equally_spaced_is_fixed_point,
    pins.test_level_fit_converged_levels_are_weighted_means,
    pins.test_level_fit_weights_equal_repetition,
    pins.test_level_fit_codes_round_trip,
    pins.test_encode_ties_go_to_the_lower_level,
    pins.test_reconstruct_round_trip,
    pins.test_reconstruct_with_codes_uses_levels,
    pins.test_level_fit_scalars_equally_spaced_is_fixed_point,
    pins.test_level_fit_scalars_converged_levels_are_means,
    pins.test_level_fit_scalars_is_unit_weight_codebook_fit,
    pins.test_codebook_grad_step_dyadic_bit_exact,
    pins.test_codebook_grad_step_quadratic_loss_gives_the_centroid,
    pins.test_levels_grad_step_dyadic_bit_exact,
    pins.test_levels_grad_step_constant_gradient_shifts_every_used_level,
]


def _failures(src_text, tmp_path, name):
    src = tmp_path / f"{name}.c"
    src.write_text(src_text)
    lib = oracle._bind(ctypes.CDLL(oracle.compile_library(str(src), str(tmp_path / f"lib{name}.so"))))
    saved = oracle._lib
    oracle._lib = lib
    failed = 0
    try:
        for pin in PINS:
            try:
                pin()
            except AssertionError:
                failed += 1
    finally:
        oracle._lib = saved
    return failed


def test_unmodified_copy_passes_every_pin(tmp_path):
    assert _failures(open(SRC).read(), tmp_path, "original") == 0


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_planted_mistake_is_caught(name, tmp_path):
    text = open(SRC).read()
    old, new = MUTANTS[name]
    assert text.count(old) == 1, f"mutation site for {name} not unique"
    assert _failures(text.replace(old, new), tmp_path, name) >= 1


def test_report_mistakes_are_caught(monkeypatch):
    # ceil(log2 k) via bit_length(k) is off by one exactly at powers of two
    monkeypatch.setattr(oracle, "ceil_log2", lambda k: k.bit_length())
    with pytest.raises(AssertionError):
        for row in pins._golden_rows():
            if row[0].startswith("table"):
                pins.test_report_tables_4_5(row)
