"""The persistent evaluation pass against the per-round launches and the oracle.

A solve without per-pass events, fingerprint or dual trace on a table whose tile-interleaved copy holds
fp32 units can run rounds 0 .. T-1 in one cooperative launch: a scenario's next round is released by
its own price update (Eq. price_update, Sec. 3.2.3) instead of a kernel boundary. It does so by default
on uniform tables with enough tiles per warp, and on request (esp_debug_set_persistent) on every table
that can take it, which is how these tests run it on small tables and sorted layouts. The arithmetic of a
round is the round pass's, so everything must be bit-identical to the per-round launches: prices and
demands after every round, selections, objectives, rounds run. The parity bar against the oracle is
the usual one (selections and demands bit-exact, prices within 1e-12 relative per step, objectives
within 1e-9 relative).
"""

import numpy as np
import pytest

import oracle
from paper_2608_07971_gb300 import esp, workloads as W

from tests.parity_util import MODES, STEPS, check_solution, rel_err

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("needs a GPU")
    from paper_2608_07971_gb300 import build
    build.build()
    esp.load_library()


def table(case):
    rng = np.random.default_rng(101)
    if case == "whatif":
        return W.whatif_batch(scenarios=[2, 9, 31, 77], J=1024).table
    if case == "heavy":
        return W.heavy_tail(scenarios=[0, 5], J=4000).table
    if case == "one_scenario":          # every physical warp shares the one scenario
        return W.cluster_512(scenarios=[3]).table
    if case == "ragged256":
        return W.random_table(rng, S=3, J=700, R=6, kmin=1, kmax=256, umax=5000)
    if case == "k1":                    # runs of single-option jobs only
        return W.random_table(rng, S=2, J=3000, R=6, kmin=1, kmax=1, umax=5000)
    if case == "r4k8":
        return W.random_table(rng, S=5, J=900, R=4, kmin=8, kmax=8, umax=5000)
    if case == "r8k32":
        return W.random_table(rng, S=2, J=600, R=8, kmin=32, kmax=32, umax=5000)
    raise ValueError(case)


def solve_both(t, eta, T, waves=0, **kw):
    a = esp.Solver()
    esp.esp_debug_set_persistent(a.ctx, 1)
    if waves:
        esp.esp_debug_set_plan_waves(a.ctx, waves)
    a.load(t)
    b = esp.Solver()
    esp.esp_debug_set_persistent(b.ctx, 0)
    if waves:
        esp.esp_debug_set_plan_waves(b.ctx, waves)
    b.load(t)
    assert esp.esp_debug_persistent(a.ctx) > 0, "the table should take the persistent pass"
    sa = a.solve(eta, T, traces="prices", **kw)
    la = a.launches()
    sb = b.solve(eta, T, traces="prices", **kw)
    lb = b.launches()
    a.close()
    b.close()
    assert la == 4, la
    assert lb == T + 3, lb
    return sa, sb


def assert_same(sa, sb):
    for f in ("lam", "sel", "demand", "lambda_trace", "demand_trace"):
        assert np.array_equal(getattr(sa, f), getattr(sb, f), equal_nan=True), f
    for f in ("rounds_run", "converged", "status", "feasible", "primal", "dual"):
        assert np.array_equal(sa.result[f], sb.result[f]), f


def check_trajectories(t, sol, eta, T, mode, step, tol=0.0, lambda0=None):
    """Final state and per-round prices and demands of every scenario against the oracle."""
    check_solution(t, sol, list(range(t.S)), eta, T, mode, step, tol=tol, lambda0=lambda0, traces=False)
    ot = oracle.OracleTable(t)
    for s in range(t.S):
        l0 = None if lambda0 is None else lambda0[s]
        ref = oracle.solve_scenario(ot, s, eta, T, mode=MODES[mode], step=STEPS[step], tol=tol, lambda0=l0,
                                    traces=True)
        n = ref.rounds_run
        assert rel_err(sol.lambda_trace[s, :n + 1], ref.lambda_trace[:n + 1]) <= 1e-12, s
        assert np.array_equal(sol.demand_trace[s, :n], ref.demand_trace[:n]), s


@pytest.mark.parametrize("case", ["whatif", "heavy", "one_scenario", "ragged256", "k1", "r4k8", "r8k32"])
def test_persistent_equals_per_round_launches(case):
    t = table(case)
    T = 40
    sa, sb = solve_both(t, 0.05, T)
    assert_same(sa, sb)
    check_trajectories(t, sa, 0.05, T, esp.ESP_PRICE_NORMALIZED, esp.ESP_STEP_FIXED)


@pytest.mark.parametrize("waves", [1, 4, 8])
def test_persistent_any_number_of_ranges_per_warp(waves):
    """Plans of 1, 4 and 8 waves of ranges (2 by default): work items of every size."""
    t = table("heavy")
    sa, sb = solve_both(t, 0.05, 30, waves=waves)
    assert_same(sa, sb)


def test_persistent_tolerance_stop():
    """Scenarios that stop at different rounds (their later rounds are released at once)."""
    t = table("ragged256")
    T = 60
    sa, sb = solve_both(t, 0.05, T, tol=0.02)
    assert_same(sa, sb)
    assert sa.result["rounds_run"].min() < T, "some scenario should stop early"
    check_trajectories(t, sa, 0.05, T, esp.ESP_PRICE_NORMALIZED, esp.ESP_STEP_FIXED, tol=0.02)


def test_persistent_warm_start_inv_sqrt_raw():
    """A warm start, the eta0/sqrt(t) step and prices in stored units."""
    t = table("whatif")
    T = 30
    l0 = np.random.default_rng(5).uniform(0.0, 2e-7, size=(t.S, t.P))
    kw = dict(mode=esp.ESP_PRICE_RAW, step=esp.ESP_STEP_INV_SQRT, lambda0=l0)
    sa, sb = solve_both(t, 2e-9, T, **kw)
    assert_same(sa, sb)
    check_trajectories(t, sa, 2e-9, T, esp.ESP_PRICE_RAW, esp.ESP_STEP_INV_SQRT, lambda0=l0)


def test_persistent_repeated_solves_and_reload():
    """The same graph replayed, then a reload of another table on the same context."""
    t1, t2 = table("whatif"), table("heavy")
    s = esp.Solver()
    esp.esp_debug_set_persistent(s.ctx, 1)
    s.load(t1)
    first = s.solve(0.05, 25, traces="prices")
    again = s.solve(0.05, 25, traces="prices")
    assert_same(first, again)
    s.load(t2)
    assert esp.esp_debug_persistent(s.ctx) > 0
    other = s.solve(0.05, 25, traces="prices")
    s.close()
    ref = esp.Solver()
    esp.esp_debug_set_persistent(ref.ctx, 0)
    ref.load(t2)
    want = ref.solve(0.05, 25, traces="prices")
    ref.close()
    assert_same(other, want)


def test_tables_that_do_not_take_it():
    """Units of 2^23 and more (fp32 would not hold them exactly), R = 5, and solves that need the
    round passes (fingerprint and dual traces, per-pass events) use the per-round launches."""
    rng = np.random.default_rng(7)
    big = W.random_table(rng, S=2, J=500, R=6, kmin=16, kmax=16, umax=1 << 24)
    r5 = W.random_table(rng, S=2, J=500, R=5, kmin=8, kmax=8, umax=5000)
    for t in (big, r5):
        s = esp.Solver()
        esp.esp_debug_set_persistent(s.ctx, 1)
        s.load(t)
        assert esp.esp_debug_persistent(s.ctx) == 0
        s.solve(0.05, 10)
        assert s.launches() == 10 + 3
        s.close()
    t = table("r4k8")
    s = esp.Solver()
    esp.esp_debug_set_persistent(s.ctx, 1)
    s.load(t)
    s.solve(0.05, 10, traces=True)
    assert s.launches() == 10 + 3
    s.solve(0.05, 10, flags=esp.ESP_FLAG_PASS_EVENTS)
    assert s.launches() == 10 + 3
    s.solve(0.05, 10)
    assert s.launches() == 4
    s.close()


def test_default_policy():
    """By default: the persistent pass on a uniform table with at least 16 tiles per warp of its launch
    (the what-if batch at 256 scenarios), one launch per round on a small uniform table and on a sorted
    layout."""
    big = W.whatif_batch(scenarios=list(range(256))).table
    small = table("whatif")
    sorted_layout = table("heavy")
    for t, want in ((big, True), (small, False), (sorted_layout, False)):
        s = esp.Solver(t)
        assert (esp.esp_debug_persistent(s.ctx) > 0) == want
        s.solve(0.02, 6)
        assert s.launches() == (4 if want else 6 + 3)
        esp.esp_debug_set_persistent(s.ctx, 0)
        assert esp.esp_debug_persistent(s.ctx) == 0
        s.solve(0.02, 6)
        assert s.launches() == 6 + 3
        s.close()
