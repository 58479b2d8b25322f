"""Shared comparison of a GPU solution with the oracle's run of the same scenarios.

The bar: selections, integer demands and selection fingerprints bit-exact; the price trajectory
within 1e-12 relative per step (bit-exact is expected: both sides perform the same IEEE operations);
primal and dual objectives within 1e-9 relative (the GPU sums in a fixed tree, the oracle in job
order).
"""

import numpy as np

import oracle
from paper_2608_07971_gb300 import esp

MODES = {esp.ESP_PRICE_RAW: oracle.RAW, esp.ESP_PRICE_NORMALIZED: oracle.NORMALIZED}
STEPS = {esp.ESP_STEP_FIXED: oracle.STEP_FIXED, esp.ESP_STEP_INV_SQRT: oracle.STEP_INV_SQRT}


def rel_err(a, b):
    a, b = np.asarray(a, np.float64), np.asarray(b, np.float64)
    den = np.maximum(np.abs(b), 1e-300)
    d = np.abs(a - b)
    return float(np.max(np.where(d == 0, 0.0, d / den))) if a.size else 0.0


def check_solution(t, sol, scen_ids, eta, T, mode, step, tol=0.0, lambda0=None, traces=True):
    """Compares GPU scenarios (rows of sol) with the oracle run of the same scenarios of t."""
    ot = oracle.OracleTable(t)
    for row, s in enumerate(scen_ids):
        l0 = None if lambda0 is None else lambda0[row]
        ref = oracle.solve_scenario(ot, s, eta, T, mode=MODES[mode], step=STEPS[step], tol=tol, lambda0=l0,
                                    traces=traces)
        check_scenario(sol, row, ref, s, traces)
    return True


def check_scenario(sol, row, ref, s, traces=True):
    """Row `row` of a GPU solution against the oracle's solution `ref` of the same scenario `s`."""
    r = sol.result[row]
    assert r["rounds_run"] == ref.rounds_run, (s, r["rounds_run"], ref.rounds_run)
    assert r["converged"] == ref.converged
    assert (r["status"] != 0) == (ref.status != 0)
    assert np.array_equal(sol.sel[row], ref.sel), f"selection differs in scenario {s}"
    assert np.array_equal(sol.demand[row], ref.demand), f"demand differs in scenario {s}"
    assert rel_err(sol.lam[row], ref.lam) <= 1e-12
    assert r["feasible"] == ref.feasible
    assert abs(r["primal"] - ref.primal) <= 1e-9 * max(1.0, abs(ref.primal))
    assert abs(r["dual"] - ref.dual) <= 1e-9 * max(1.0, abs(ref.dual))
    if traces:
        n = ref.rounds_run
        assert rel_err(sol.lambda_trace[row, :n + 1], ref.lambda_trace[:n + 1]) <= 1e-12
        assert np.array_equal(sol.demand_trace[row, :n], ref.demand_trace[:n]), f"U^t differs in {s}"
        assert np.array_equal(sol.selhash_trace[row, :n], ref.selhash_trace[:n]), f"hash differs in {s}"
        assert rel_err(sol.dual_trace[row, :n + 1], ref.dual_trace[:n + 1]) <= 1e-9
        assert abs(r["best_dual"] - ref.best_dual) <= 1e-9 * max(1.0, abs(ref.best_dual))
    return True
