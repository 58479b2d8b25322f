"""The pins are strong enough: each plausible mistake planted in a temporary copy of the oracle
(a dropped term, a wrong sign, a transposed index, a wrong tie rule, ...) fails at least one pin.
Mistakes are planted on the CPU only, in a copy compiled to a temporary directory."""

import os
import shutil
import subprocess

import numpy as np
import pytest

import oracle
from tests import test_oracle_penalties as pen
from tests import test_oracle_pins as pins

SRC = os.path.join(os.path.dirname(oracle.__file__), "esp_oracle.c")

MUTANTS = {
    "tie_to_highest_index": ("if (score < best_score) {", "if (score <= best_score) {"),
    "value_sign": ("double score = -t->values[o];", "double score = t->values[o];"),
    "dropped_last_column": ("    for (int32_t r = 0; r < t->R; ++r) {\n        double price",
                            "    for (int32_t r = 0; r < t->R - 1; ++r) {\n        double price"),
    "reversed_price_columns": ("p[esp_oracle_price_index(t, o, r)]", "p[esp_oracle_price_index(t, o, t->R - 1 - r)]"),
    "update_sign": ("fma(eta, excess, lambda_in[k])", "fma(-eta, excess, lambda_in[k])"),
    "no_projection": ("moved > 0.0 ? moved : 0.0", "moved"),
    "normalized_not_divided": ("            excess = excess / (double)cap[k];", "            excess = excess;"),
    "step_index_off_by_one": ("eta = prm->eta0 / sqrt((double)t1);", "eta = prm->eta0 / sqrt((double)(t1 + 1));"),
    "dual_without_capacity": ("g += lambda[k] * (double)cap[k];", "g += lambda[k];"),
    "group_stride": ("(t->R - t->r_global) * (int32_t)t->group[o]", "(int32_t)t->group[o]"),
    "effective_price_not_normalized": ("p[k] = lambda[k] / (double)cap[k];", "p[k] = lambda[k];"),
    "convergence_strict": ("converged = delta <= prm->tol * scale;", "converged = delta < prm->tol * scale;"),
    "demand_wrong_column": ("demand[esp_oracle_price_index(t, best, r)] +=", "demand[r % t->P] +="),
    "primal_first_option": ("primal += t->values[t->job_off[(int64_t)s * J + j] + sel[j]];",
                            "primal += t->values[t->job_off[(int64_t)s * J + j]];"),
    "switching_cost_inverted": ("(c_cur >= 0 && c != c_cur) ? gamma0", "(c_cur >= 0 && c == c_cur) ? gamma0"),
    "interference_not_clamped": ("    if (excess < 0.0)\n        excess = 0.0;\n", ""),
    "penalty_added_to_value": ("values_out[o] = t->values[o] - gamma;", "values_out[o] = t->values[o] + gamma;"),
    "threshold_not_clamped": ("    if (add > beta_max)\n        add = beta_max;\n", ""),
    "capacity_largest_footprint": ("if (q_units[o * R + r] < m)", "if (q_units[o * R + r] > m)"),
    "best_dual_tracks_largest": ("        if (g < best_dual)\n            best_dual = g;\n        if (dual_trace)\n            dual_trace[it] = g;",
                                 "        if (g > best_dual || best_dual == INFINITY)\n            best_dual = g;\n        if (dual_trace)\n            dual_trace[it] = g;"),
    "feasible_only_below_capacity": ("if (demand[k] > cap[k])", "if (demand[k] >= cap[k])"),
    "stopping_scale_from_new_prices": ("if (fabs(lambda[k]) > scale)\n                    scale = fabs(lambda[k]);",
                                       "if (fabs(next[k]) > scale)\n                    scale = fabs(next[k]);"),
}


def pin_suite():
    """Every pin, with fixed parameters. Each call raises AssertionError on a mismatch."""
    yield pins.test_two_job_cycle_matches_hand_trajectory
    for seed in range(3):
        for mode in (oracle.RAW, oracle.NORMALIZED):
            yield lambda seed=seed, mode=mode: pins.test_weak_duality_every_round_against_brute_force(seed, mode)
    yield pins.test_primal_is_sum_of_selected_values
    for seed in range(2):
        for groups in (0, 3):
            yield lambda seed=seed, groups=groups: pins.test_best_response_is_exact_argmin_within_rounding(seed, groups)
        yield lambda seed=seed: pins.test_best_response_bit_exact_on_dyadic_inputs_with_ties(seed)
    yield pins.test_zero_prices_pick_largest_value_lowest_index
    yield pins.test_capacity_never_binding_keeps_prices_zero
    yield pins.test_single_resource_two_option_switch_price
    yield pins.test_identical_options_select_index_zero
    for mode in (oracle.RAW, oracle.NORMALIZED):
        for step in (oracle.STEP_FIXED, oracle.STEP_INV_SQRT):
            yield lambda mode=mode, step=step: pins.test_constant_excess_closed_form(mode, step)
            yield lambda mode=mode, step=step: pins.test_invariants_tiny_cluster(mode, step)
    yield pins.test_projection_clamps_at_zero
    yield lambda: pins.test_invariants_random_grouped(0)
    yield pins.test_fixed_point_complementary_slackness
    yield pins.test_tolerance_stops_early_and_freezes
    yield pins.test_tolerance_rule_boundary_is_inclusive
    yield pins.test_tolerance_scale_is_the_current_price
    yield pins.test_scenarios_are_independent
    yield pins.test_warm_start_resumes_the_trajectory
    yield pen.test_adaptive_threshold_closed_form
    yield pen.test_switching_cost_shifts_switch_price
    yield pen.test_interference_penalty_only_above_threshold
    yield pen.test_large_switching_cost_keeps_current_configuration
    yield pen.test_effective_capacity_hand_example


def failing_pins(lib):
    saved = dict(oracle._lib_cache)
    real_load = oracle.load
    oracle.load = lambda path=None: lib
    failures = 0
    try:
        for pin in pin_suite():
            try:
                pin()
            except (AssertionError, ValueError, IndexError, OverflowError, ZeroDivisionError):
                failures += 1
    finally:
        oracle.load = real_load
        oracle._lib_cache.clear()
        oracle._lib_cache.update(saved)
    return failures


def test_unmodified_oracle_passes_every_pin():
    assert failing_pins(oracle.load()) == 0


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_planted_mistake_is_caught(name, tmp_path):
    old, new = MUTANTS[name]
    src = open(SRC).read()
    assert src.count(old) >= 1, f"mutation anchor missing: {name}"
    mutant = tmp_path / "esp_oracle.c"
    mutant.write_text(src.replace(old, new))
    shutil.copy(os.path.join(os.path.dirname(SRC), "esp_oracle.h"), tmp_path / "esp_oracle.h")
    so = tmp_path / "liboracle_mutant.so"
    subprocess.check_call(["gcc", *oracle.CFLAGS, str(mutant), "-o", str(so), "-lm"])
    oracle._lib_cache.pop(str(so), None)
    lib = oracle.load(str(so))
    with np.errstate(all="ignore"):
        assert failing_pins(lib) > 0, f"no pin caught mutant {name}"
