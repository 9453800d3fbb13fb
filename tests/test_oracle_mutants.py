"""The pins are strong enough: plant a plausible mistake in a copy of the oracle
source (a dropped term, a wrong sign or index, a transposed operand, a wrong
tie rule), build it, and check that at least one pin fails.

Mistakes are planted only in temporary copies of ``oracle/qe_oracle.c``, on the
CPU; the committed oracle is never modified.
"""
import os
import subprocess

import numpy as np
import pytest

import oracle
import tests.test_oracle_golden as golden
import tests.test_oracle_pins as pins

# (name, text in qe_oracle.c, planted replacement)
MUTANTS = [
    ("beta_sign", "double b = -u;", "double b = u;"),
    ("drop_diag_term", "double u = (WS[j] - djj * Wh[j] - TS[j]) / djj;",
     "double u = (WS[j] - TS[j]) / djj;"),
    ("skip_rank1_part_A", "WS[k] -= old * Sj[k];", "WS[k] -= 0.0 * Sj[k];"),
    ("truncate_not_round", "double c = nearbyint(x / s + z);", "double c = floor(x / s + z);"),
    ("zero_point_sign", "float z = nearbyintf(-lo / s);", "float z = nearbyintf(lo / s);"),
    ("grid_no_zero_in_range", "float lo = 0.0f, hi = 0.0f;", "float lo = 1e30f, hi = -1e30f;"),
    ("sigma_wrong_operand", "acc += X[a * n + k] * X[b * n + k];", "acc += X[a * n + k] * X[a * n + k];"),
    ("alg3_P_after_zero_diag", "acc += Wi[k] * Sn[k * p + j];", "if (k != j) acc += Wi[k] * Sn[k * p + j];"),
    ("alg3_drop_last_term", "for (int64_t k = 0; k < j; ++k)   /* k = j adds Sn_jj = 0 */",
     "for (int64_t k = 0; k + 1 < j; ++k)"),
    ("objective_wrong_index", "t += Sa[b] * d[b];", "t += Sa[b] * d[a];"),
    ("topk_reversed_ties", "if (x->idx < y->idx) return -1;      /* tie: smaller linear index first */",
     "if (x->idx < y->idx) return 1;"),
    ("iht_wrong_step_sign", "T[i * p + j] = H[i * p + j] - eta * 2.0 * G[j];",
     "T[i * p + j] = H[i * p + j] + eta * 2.0 * G[j];"),
    ("iht_step_wrong_sign", "T[i * p + j] = H[i * p + j] - 2.0 * eta * G[j];",
     "T[i * p + j] = H[i * p + j] + 2.0 * eta * G[j];"),
    ("iht_step_target_not_level", "D[j] = H[i * p + j] + qo_level(codes[i * p + j], scale[i], zero[i]) - W[i * p + j];",
     "D[j] = H[i * p + j] + W[i * p + j] - W[i * p + j];"),
    ("power_wrong_rayleigh", "lam += v[a] * w[a];", "lam += w[a] * w[a];"),
    ("column_norm_not_squared", "norm2[j] += T[i * p + j] * T[i * p + j];", "norm2[j] += T[i * p + j];"),
    ("relax_keeps_level", "                Wh[j] = b;\n", "                Wh[j] = qo_level(c, s, z);\n"),
    ("relax_last_sweep_too", "t1 % relax_period == 0 && t1 < iters;", "t1 % relax_period == 0 && t1 <= iters;"),
    ("group_scale_of_first_group", "const double s = srow[j / gsize], z = zrow[j / gsize];",
     "const double s = srow[0], z = zrow[0];"),
    ("group_range_from_row_start", "for (int64_t j = g * gsize; j < j1; ++j) {", "for (int64_t j = 0; j < j1; ++j) {"),
]

PINS = [
    lambda: pins.test_quantizer_returns_nearest_level(3),
    lambda: pins.test_grid_covers_row_range_and_zero(3),
    lambda: pins.test_every_update_is_bruteforce_argmin(3),
    lambda: pins.test_exhaustive_tiny_layer_cw_minimum(3),
    lambda: pins.test_objective_non_increasing(1, True),
    lambda: pins.test_algorithm1_equals_algorithm3(4, 0),
    pins.test_diagonal_sigma_gives_round_to_nearest,
    pins.test_objective_matches_direct_residual,
    pins.test_sigma_properties,
    pins.test_power_lambda_matches_eigvalsh,
    pins.test_topk_matches_full_sort_with_ties,
    pins.test_outlier_iht_descent_and_budget,
    pins.test_column_selection_is_the_projection,
    pins.test_structured_outlier_descent_budget_and_columns,
    lambda: pins.test_relaxed_sweep_is_one_gauss_seidel_step(3),
    pins.test_relaxed_sweeps_converge_to_w,
    pins.test_relax_period_not_below_iters_is_plain_algorithm1,
    lambda: pins.test_grouped_grid_is_the_row_rule_per_group(3, 16),
    pins.test_grouped_diagonal_sigma_gives_per_group_round_to_nearest,
    lambda: pins.test_grouped_update_is_bruteforce_argmin_on_its_group(2),
    golden.test_hand_worked_two_feature_layer,
    lambda: pins.test_iht_step_gradient_and_projection(False),
    pins.test_iht_step_replays_algorithm4,
]


@pytest.mark.parametrize("name,old,new", MUTANTS, ids=[m[0] for m in MUTANTS])
def test_planted_mistake_is_caught(name, old, new, tmp_path, monkeypatch):
    src = open(oracle.SRC).read()
    assert src.count(old) == 1, f"mutation anchor for {name} not unique"
    mutant_src = tmp_path / f"qe_oracle_{name}.c"
    mutant_src.write_text(src.replace(old, new))
    lib = oracle.build(str(mutant_src), str(tmp_path / f"lib_{name}.so"), force=True)
    mutant = oracle.Oracle(lib)
    monkeypatch.setattr(pins, "O", mutant)
    monkeypatch.setattr(golden, "O", mutant)
    caught = []
    for pin in PINS:
        try:
            with np.errstate(all="ignore"):
                pin()
        except (AssertionError, ValueError, FloatingPointError, IndexError, KeyError):
            caught.append(pin)
    assert caught, f"no pin caught the planted mistake {name}"
