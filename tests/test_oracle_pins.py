"""Pins for the oracle of the ESP tatonnement (Sec. 3.2): checks against things other than the oracle.

- a hand-worked two-job trajectory in exact dyadic arithmetic (tests/golden/two_job_cycle.json);
- brute force over every joint selection of tiny integer programs (Eqs. primal_obj..integer), with
  weak duality of g(lambda) (Eq. lagrangian) checked in exact rational arithmetic at every round;
- per-job best responses against exact rational reduced costs (exact argmin within the fp64
  rounding bound; bit-exact with the lowest-index tie rule on dyadic inputs);
- closed forms (lambda = 0, never-binding capacity, the R=1 K=2 switch price, constant excess under
  both step rules and both price units) and the invariants of Eq. price_update along trajectories;
- complementary slackness at a constructed fixed point.
"""

import itertools
import json
import math
import os
from fractions import Fraction

import numpy as np
import pytest

import oracle
from paper_2608_07971_gb300 import workloads as W

HERE = os.path.dirname(os.path.abspath(__file__))
EPS = 2.0 ** -53


def table_from_jobs(jobs, capacity, R=None, group=None, r_global=None, P=None):
    """jobs: list of lists of (value, units-tuple). One scenario."""
    R = R or len(jobs[0][0][1])
    K = [len(j) for j in jobs]
    off = np.zeros(len(jobs) + 1, np.int64)
    off[1:] = np.cumsum(K)
    units = np.array([u for j in jobs for (_, u) in j], np.int32).reshape(-1, R)
    values = np.array([v for j in jobs for (v, _) in j], np.float64)
    cap = np.asarray(capacity, np.int64).reshape(1, -1)
    P = P or cap.shape[1]
    return W.OptionTable(1, len(jobs), R, P, R if r_global is None else r_global, off, units,
                         values, None if group is None else np.asarray(group, np.uint16), cap)


def price_col(t, o, r):
    """Priced resource of stored column r of option o (the table's own definition)."""
    if t.group is None or r < t.r_global:
        return r
    return t.r_global + (t.R - t.r_global) * int(t.group[o]) + (r - t.r_global)


def exact_scores(t, s, p):
    """Exact rational reduced cost -v + sum_r p * u of every option of scenario s."""
    pf = [x if isinstance(x, Fraction) else Fraction(float(x)) for x in p]
    out = []
    for j in range(t.J):
        a, b = int(t.job_off[s * t.J + j]), int(t.job_off[s * t.J + j + 1])
        out.append([-Fraction(float(t.values[o])) +
                    sum(pf[price_col(t, o, r)] * int(t.units[o, r]) for r in range(t.R))
                    for o in range(a, b)])
    return out


def magnitude(t, o, p):
    return abs(float(t.values[o])) + sum(float(p[price_col(t, o, r)]) * int(t.units[o, r]) for r in range(t.R))


def brute_force_opt(t, s=0):
    """max sum v subject to capacity over all prod K_j joint selections (exact)."""
    best, arg = None, None
    ranges = [range(int(t.job_off[s * t.J + j + 1] - t.job_off[s * t.J + j])) for j in range(t.J)]
    for choice in itertools.product(*ranges):
        use = [0] * t.P
        val = Fraction(0)
        for j, c in enumerate(choice):
            o = int(t.job_off[s * t.J + j]) + c
            val += Fraction(float(t.values[o]))
            for r in range(t.R):
                use[price_col(t, o, r)] += int(t.units[o, r])
        if all(use[k] <= int(t.capacity[s, k]) for k in range(t.P)) and (best is None or val > best):
            best, arg = val, choice
    return best, arg


def exact_dual(t, s, p):
    """g at multiplier p (the effective per-unit price): sum_j max_c (v - p.u) + sum_k p_k C_k."""
    sc = exact_scores(t, s, p)
    pf = [x if isinstance(x, Fraction) else Fraction(float(x)) for x in p]
    return sum(-min(js) for js in sc) + sum(pf[k] * int(t.capacity[s, k]) for k in range(t.P))


# ---------------------------------------------------------------------------------------------
# Hand-worked trajectory


def load_golden():
    with open(os.path.join(HERE, "golden", "two_job_cycle.json")) as f:
        return json.load(f)


def test_two_job_cycle_matches_hand_trajectory():
    g = load_golden()
    inst = g["instance"]
    jobs = [[(o["value"], (o["units"],)) for o in j["options"]] for j in inst["jobs"]]
    t = table_from_jobs(jobs, [inst["capacity"]])
    T = len(g["hand_trajectory"]) - 1
    sol = oracle.solve_scenario(t, 0, float(Fraction(inst["eta0"])), T, mode=oracle.RAW,
                                traces=True, sel_trace=True)
    for row in g["hand_trajectory"][:T]:
        ti = row["t"]
        assert sol.lambda_trace[ti, 0] == float(Fraction(row["lambda"])), ti
        assert sol.sel_trace[ti].tolist() == row["selection"], ti
        assert sol.demand_trace[ti, 0] == row["demand"], ti
        assert sol.dual_trace[ti] == float(Fraction(row["dual"])), ti
    last = g["hand_trajectory"][T]
    assert sol.lambda_trace[T, 0] == float(Fraction(last["lambda"]))
    assert sol.lam[0] == float(Fraction(last["lambda"]))
    assert sol.sel.tolist() == last["selection"]
    assert sol.demand[0] == last["demand"]
    assert sol.rounds_run == T
    # weak duality against the hand IP optimum, and the best dual is the smallest g seen
    opt = Fraction(g["ip_optimum"]["value"])
    assert all(Fraction(x) >= opt for x in sol.dual_trace)
    assert sol.best_dual == min(sol.dual_trace)
    assert brute_force_opt(t)[0] == opt
    assert brute_force_opt(t)[1] == tuple(g["ip_optimum"]["selection"])
    lp = Fraction(g["lp_bound"]["value"])
    assert exact_dual(t, 0, [Fraction(g["lp_bound"]["at_lambda"])]) == lp


# ---------------------------------------------------------------------------------------------
# Brute force and weak duality


@pytest.mark.parametrize("mode", [oracle.RAW, oracle.NORMALIZED])
@pytest.mark.parametrize("seed", range(6))
def test_weak_duality_every_round_against_brute_force(seed, mode):
    rng = np.random.default_rng(100 + seed)
    t = W.random_table(rng, S=1, J=int(rng.integers(2, 6)), R=int(rng.integers(1, 4)), kmin=1, kmax=4,
                       umax=20, cap_frac=0.6)
    opt, _ = brute_force_opt(t)
    eta = 0.01 if mode == oracle.RAW else 0.3
    sol = oracle.solve_scenario(t, 0, eta, 40, mode=mode, traces=True)
    for ti in range(sol.rounds_run + 1):
        lam = sol.lambda_trace[ti]
        p = oracle.effective_prices(t, 0, lam, mode)
        g_exact = exact_dual(t, 0, p)
        if opt is not None:
            assert g_exact >= opt, (ti, float(g_exact), float(opt))
        # the oracle's g agrees with the exact value up to fp64 rounding of the sums
        scale = sum(abs(float(v)) for v in t.values) + float(np.sum(lam * t.capacity[0])) + 1.0
        assert abs(float(g_exact) - sol.dual_trace[ti]) <= 1e-12 * scale
    if sol.feasible and opt is not None:
        assert Fraction(sol.primal) <= opt + Fraction(1, 10**9)


def test_primal_is_sum_of_selected_values():
    rng = np.random.default_rng(7)
    t = W.random_table(rng, S=1, J=30, R=3, kmin=1, kmax=6)
    sol = oracle.solve_scenario(t, 0, 0.2, 25)
    picked = t.job_off[:-1] + sol.sel
    assert sol.primal == pytest.approx(float(np.sum(t.values[picked])), rel=1e-14)
    assert sol.demand.tolist() == t.units[picked].sum(axis=0).tolist()
    assert sol.feasible == int(np.all(sol.demand <= t.capacity[0]))


# ---------------------------------------------------------------------------------------------
# Best response against exact arithmetic


@pytest.mark.parametrize("groups", [0, 3])
@pytest.mark.parametrize("seed", range(5))
def test_best_response_is_exact_argmin_within_rounding(seed, groups):
    rng = np.random.default_rng(200 + seed)
    t = W.random_table(rng, S=2, J=12, R=4, kmin=1, kmax=7, umax=1000, groups=groups,
                       r_global=2 if groups else None)
    for s in range(t.S):
        lam = rng.exponential(1e-3, size=t.P)
        lam[rng.random(t.P) < 0.2] = 0.0
        for mode in (oracle.RAW, oracle.NORMALIZED):
            p = oracle.effective_prices(t, s, lam, mode)
            want_p = lam if mode == oracle.RAW else lam / t.capacity[s]
            assert np.array_equal(p, want_p)
            sel, dem, ms = oracle.best_response(t, s, lam, mode)
            sc = exact_scores(t, s, p)
            for j in range(t.J):
                a = int(t.job_off[s * t.J + j])
                o = a + int(sel[j])
                bound = 2 * t.R * EPS * max(magnitude(t, a + c, p) for c in range(len(sc[j])))
                assert float(sc[j][sel[j]] - min(sc[j])) <= bound
                assert abs(float(sc[j][sel[j]]) - ms[j]) <= bound
            picked = t.job_off[s * t.J:(s + 1) * t.J] + sel
            want = np.zeros(t.P, np.int64)
            for o in picked:
                for r in range(t.R):
                    want[price_col(t, o, r)] += int(t.units[o, r])
            assert dem.tolist() == want.tolist()


@pytest.mark.parametrize("seed", range(5))
def test_best_response_bit_exact_on_dyadic_inputs_with_ties(seed):
    rng = np.random.default_rng(300 + seed)
    t = W.random_table(rng, S=1, J=40, R=3, kmin=1, kmax=6, umax=12, dyadic=True)
    # duplicate some options so exact ties occur
    for j in range(0, t.J, 3):
        a, b = int(t.job_off[j]), int(t.job_off[j + 1])
        if b - a >= 2:
            t.units[b - 1] = t.units[a]
            t.values[b - 1] = t.values[a]
    lam = rng.integers(0, 8, size=t.P) / 64.0
    sel, dem, ms = oracle.best_response(t, 0, lam, oracle.RAW)
    sc = exact_scores(t, 0, lam)
    for j in range(t.J):
        m = min(sc[j])
        assert sel[j] == sc[j].index(m)           # lowest index among exact minima
        assert ms[j] == float(m)                   # exact, no rounding on dyadic data


# ---------------------------------------------------------------------------------------------
# Special cases and closed forms


def test_zero_prices_pick_largest_value_lowest_index():
    rng = np.random.default_rng(11)
    t = W.random_table(rng, S=1, J=25, R=2, kmin=1, kmax=6, dyadic=True)
    sel, _, ms = oracle.best_response(t, 0, np.zeros(t.P), oracle.RAW)
    for j in range(t.J):
        v = t.values[t.job_off[j]:t.job_off[j + 1]]
        assert sel[j] == int(np.argmax(v))        # numpy argmax returns the first maximum
        assert ms[j] == -v.max()


def test_capacity_never_binding_keeps_prices_zero():
    rng = np.random.default_rng(12)
    t = W.random_table(rng, S=1, J=10, R=3, kmin=2, kmax=5)
    t.capacity[:] = 10**12
    sol = oracle.solve_scenario(t, 0, 0.5, 30, mode=oracle.RAW, traces=True)
    assert np.all(sol.lambda_trace == 0.0)
    for j in range(t.J):
        assert sol.sel[j] == int(np.argmax(t.values[t.job_off[j]:t.job_off[j + 1]]))


def test_single_resource_two_option_switch_price():
    # (v, u) = (5, 10) and (2, 4): the rents equalise at lambda* = (5 - 2) / (10 - 4) = 1/2
    t = table_from_jobs([[(5.0, (10,)), (2.0, (4,))]], [100])
    lam_star = 0.5
    for lam, want in [(lam_star - 2**-20, 0), (lam_star, 0), (lam_star + 2**-20, 1), (0.0, 0), (10.0, 1)]:
        sel, _, ms = oracle.best_response(t, 0, np.array([lam]), oracle.RAW)
        assert sel[0] == want, lam
    sel, _, ms = oracle.best_response(t, 0, np.array([lam_star]), oracle.RAW)
    assert ms[0] == 0.0


def test_identical_options_select_index_zero():
    t = table_from_jobs([[(1.5, (3, 4))] * 5, [(0.25, (1, 0))] * 3], [10, 10])
    for lam in (np.zeros(2), np.array([0.1, 7.0]), np.array([3.0, 0.0])):
        sel, _, _ = oracle.best_response(t, 0, lam, oracle.RAW)
        assert sel.tolist() == [0, 0]


@pytest.mark.parametrize("mode", [oracle.RAW, oracle.NORMALIZED])
@pytest.mark.parametrize("step", [oracle.STEP_FIXED, oracle.STEP_INV_SQRT])
def test_constant_excess_closed_form(mode, step):
    # one job, one option using C + d: U - C = d every round, so
    # lambda^T = eta0 * e * sum_{t=1..T} w_t with e = d (RAW) or d / C (NORMALIZED), w_t = 1 or 1/sqrt(t)
    C, d, eta, T = 64, 24, 0.125, 50
    t = table_from_jobs([[(1.0, (C + d,))]], [C])
    sol = oracle.solve_scenario(t, 0, eta, T, mode=mode, step=step, traces=True)
    e = d if mode == oracle.RAW else d / C
    for ti in range(T + 1):
        w = ti if step == oracle.STEP_FIXED else sum(1.0 / math.sqrt(k) for k in range(1, ti + 1))
        want = eta * e * w
        assert sol.lambda_trace[ti, 0] == pytest.approx(want, rel=4 * (ti + 1) * EPS, abs=0.0)
    if step == oracle.STEP_FIXED:                  # dyadic: exact
        assert sol.lam[0] == eta * e * T


def test_projection_clamps_at_zero():
    # demand below capacity from lambda = 0 keeps lambda at exactly 0 (never negative)
    t = table_from_jobs([[(1.0, (3,)), (2.0, (5,))]], [100])
    sol = oracle.solve_scenario(t, 0, 1.0, 5, mode=oracle.RAW, traces=True)
    assert np.all(sol.lambda_trace == 0.0)
    lam0 = np.array([3.0])   # 3 + 1 * (5 - 100) < 0 -> 0
    sol = oracle.solve_scenario(t, 0, 1.0, 3, mode=oracle.RAW, lambda0=lam0, traces=True)
    assert sol.lambda_trace[1, 0] == 0.0


def test_nonfinite_price_is_reported():
    t = table_from_jobs([[(1.0, (2**30,))]], [1])
    sol = oracle.solve_scenario(t, 0, 1e300, 5, mode=oracle.RAW)
    assert sol.status == 2
    assert sol.rounds_run == 0


# ---------------------------------------------------------------------------------------------
# Invariants along trajectories


def splitmix64(z):
    z &= (1 << 64) - 1
    z = ((z ^ (z >> 30)) * 0xBF58476D1CE4E5B9) & ((1 << 64) - 1)
    z = ((z ^ (z >> 27)) * 0x94D049BB133111EB) & ((1 << 64) - 1)
    return z ^ (z >> 31)


def check_trajectory_invariants(t, s, sol, eta, mode, step):
    J, P = t.J, t.P
    cap = t.capacity[s]
    base = t.job_off[s * J:(s + 1) * J]
    for ti in range(sol.rounds_run):
        lam, nxt = sol.lambda_trace[ti], sol.lambda_trace[ti + 1]
        assert np.all(lam >= 0.0) and np.all(nxt >= 0.0)
        U = sol.demand_trace[ti]
        # U^t recomputed from the selections
        picked = base + sol.sel_trace[ti]
        want = np.zeros(P, np.int64)
        for o in picked:
            for r in range(t.R):
                want[price_col(t, o, r)] += int(t.units[o, r])
        assert U.tolist() == want.tolist()
        # sign of the move follows the excess demand; a clamp only where the step would go below 0
        up, down = nxt > lam, nxt < lam
        assert np.all(U[up] > cap[up])
        assert np.all(U[down] < cap[down])
        clamped = (nxt == 0.0) & (lam > 0.0)
        assert np.all(U[clamped] < cap[clamped])
        # selection fingerprint
        h = sum(splitmix64((j << 32) | int(c)) for j, c in enumerate(sol.sel_trace[ti])) & ((1 << 64) - 1)
        assert int(sol.selhash_trace[ti]) == h
    assert sol.best_dual == pytest.approx(np.nanmin(sol.dual_trace[:sol.rounds_run + 1]), rel=0, abs=0)
    if sol.feasible:
        assert np.all(sol.dual_trace[:sol.rounds_run + 1] >= sol.primal - 1e-9 * (1 + abs(sol.primal)))


@pytest.mark.parametrize("mode", [oracle.RAW, oracle.NORMALIZED])
@pytest.mark.parametrize("step", [oracle.STEP_FIXED, oracle.STEP_INV_SQRT])
def test_invariants_tiny_cluster(mode, step):
    w = W.tiny_cluster()
    eta = w.eta0 if mode == oracle.NORMALIZED else 1e-7
    sol = oracle.solve_scenario(w.table, 0, eta, 200, mode=mode, step=step, traces=True, sel_trace=True)
    assert sol.status == 0 and sol.rounds_run == 200
    check_trajectory_invariants(w.table, 0, sol, eta, mode, step)


@pytest.mark.parametrize("seed", range(4))
def test_invariants_random_grouped(seed):
    rng = np.random.default_rng(400 + seed)
    t = W.random_table(rng, S=1, J=50, R=5, kmin=1, kmax=9, groups=4, r_global=3)
    sol = oracle.solve_scenario(t, 0, 0.05, 60, mode=oracle.NORMALIZED, traces=True, sel_trace=True)
    check_trajectory_invariants(t, 0, sol, 0.05, oracle.NORMALIZED, oracle.STEP_FIXED)


# ---------------------------------------------------------------------------------------------
# Convergence and complementary slackness


def test_fixed_point_complementary_slackness():
    # one job: (10, 8) or (4, 5); C = 5; raw prices, eta = 1/8. lambda climbs by 3/8 while the
    # large option is chosen; at lambda = 9/4 the small one wins (29/4 < 8), U = C and lambda stays.
    # Resource 2 never binds, so its price stays 0 with U < C.
    t = table_from_jobs([[(10.0, (8, 1)), (4.0, (5, 1))]], [5, 100])
    sol = oracle.solve_scenario(t, 0, 0.125, 100, mode=oracle.RAW, tol=1e-12, traces=True)
    assert sol.converged == 1
    assert sol.rounds_run == 7
    assert sol.lam.tolist() == [2.25, 0.0]
    assert sol.sel.tolist() == [1]
    assert sol.demand.tolist() == [5, 1]
    for k in range(2):     # lambda_k > 0 => U_k = C_k ; U_k < C_k => lambda_k = 0
        if sol.lam[k] > 0:
            assert sol.demand[k] == t.capacity[0, k]
        if sol.demand[k] < t.capacity[0, k]:
            assert sol.lam[k] == 0.0
    assert sol.primal == 4.0 and sol.feasible == 1


def test_tolerance_stops_early_and_freezes():
    w = W.tiny_cluster()
    full = oracle.solve_scenario(w.table, 0, 0.05, 200, mode=oracle.NORMALIZED, step=oracle.STEP_INV_SQRT,
                                 traces=True)
    ratio = [np.max(np.abs(full.lambda_trace[t] - full.lambda_trace[t - 1])) /
             max(1.0, np.max(np.abs(full.lambda_trace[t - 1]))) for t in range(1, 201)]
    tol = float(np.median(ratio))
    early = oracle.solve_scenario(w.table, 0, 0.05, 200, mode=oracle.NORMALIZED, step=oracle.STEP_INV_SQRT,
                                  tol=tol, traces=True)
    n = early.rounds_run
    assert early.converged == 1 and n < 200
    assert n == 1 + next(i for i, r in enumerate(ratio) if r <= tol)
    # identical prefix; the frozen prices are the ones of update n
    assert np.array_equal(early.lambda_trace[:n + 1], full.lambda_trace[:n + 1])
    assert np.array_equal(early.lam, full.lambda_trace[n])


def test_tolerance_rule_boundary_is_inclusive():
    # constant excess d = 8 at eta = 1/256 (raw): every update moves lambda by exactly 1/32 while
    # lambda <= 1 keeps the scale max(1, |lambda|) at 1. tol = 1/32 stops after the first update;
    # a slightly smaller tol never stops.
    t = table_from_jobs([[(1.0, (72,))]], [64])
    sol = oracle.solve_scenario(t, 0, 1.0 / 256, 20, mode=oracle.RAW, tol=1.0 / 32)
    assert sol.converged == 1 and sol.rounds_run == 1 and sol.lam[0] == 1.0 / 32
    sol = oracle.solve_scenario(t, 0, 1.0 / 256, 20, mode=oracle.RAW, tol=1.0 / 32 - 2**-40)
    assert sol.converged == 0 and sol.rounds_run == 20 and sol.lam[0] == 20.0 / 32


def test_tolerance_scale_is_the_current_price():
    # the stopping rule compares the move with tol * max(1, |lambda^t|), the prices before the
    # update. Constant excess d = 2 at eta = 1/2 (raw): lambda^t = t, every move is 1. With tol = 1/8
    # the move reaches the threshold once lambda^t = 8, so the update from 8 to 9 is the last (9
    # updates); scaling by the new prices instead would stop one update earlier.
    t = table_from_jobs([[(1.0, (12,))]], [10])
    sol = oracle.solve_scenario(t, 0, 0.5, 50, mode=oracle.RAW, tol=0.125)
    assert sol.converged == 1 and sol.rounds_run == 9 and sol.lam[0] == 9.0


def test_scenarios_are_independent():
    """Scenario s of a batch solves exactly as the same scenario alone (offsets re-based to 0), with
    capacities that differ between scenarios, so that any mistake in the per-scenario offsets of
    the capacities, prices or options changes the result."""
    rng = np.random.default_rng(61)
    t = W.random_table(rng, S=3, J=25, R=3, kmin=1, kmax=6, cap_frac=0.5)
    cap = t.capacity.copy()
    cap[1] = cap[1] * 100                  # never binding: feasible
    cap[2] = np.maximum(1, cap[2] // 3)
    t = W.OptionTable(**{**t.__dict__, "capacity": cap})
    flags = set()
    for mode in (oracle.RAW, oracle.NORMALIZED):
        eta = 0.002 if mode == oracle.RAW else 0.3
        for s in range(t.S):
            a = oracle.solve_scenario(t, s, eta, 30, mode=mode, traces=True)
            b = oracle.solve_scenario(t.scenario(s), 0, eta, 30, mode=mode, traces=True)
            for f in ("lam", "sel", "demand", "min_score", "lambda_trace", "demand_trace", "dual_trace"):
                assert np.array_equal(getattr(a, f), getattr(b, f)), (mode, s, f)
            assert (a.primal, a.dual, a.best_dual, a.feasible) == (b.primal, b.dual, b.best_dual, b.feasible)
            assert a.feasible == int(np.all(a.demand <= cap[s]))
            flags.add((s, a.feasible, int(np.all(a.demand <= cap[0]))))
    # some scenario is feasible under its own capacities and not under scenario 0's, or the reverse
    assert any(own != first for _, own, first in flags), flags
    # the scenarios do differ
    assert not np.array_equal(oracle.solve_scenario(t, 1, 0.3, 30).lam, oracle.solve_scenario(t, 2, 0.3, 30).lam)


def test_warm_start_resumes_the_trajectory():
    """With a fixed step, T1 updates followed by T2 more from the prices reached (lambda0) are the
    trajectory of T1 + T2 updates; the solve's minimal reduced costs are those of a best response at
    its final prices."""
    rng = np.random.default_rng(62)
    t = W.random_table(rng, S=1, J=30, R=4, kmin=1, kmax=7, cap_frac=0.4)
    full = oracle.solve_scenario(t, 0, 0.25, 24, traces=True)
    head = oracle.solve_scenario(t, 0, 0.25, 10)
    tail = oracle.solve_scenario(t, 0, 0.25, 14, lambda0=head.lam, traces=True)
    assert np.array_equal(tail.lam, full.lam) and np.array_equal(tail.sel, full.sel)
    assert np.array_equal(tail.lambda_trace, full.lambda_trace[10:])
    assert np.array_equal(tail.demand_trace, full.demand_trace[10:])
    assert len(np.unique(full.lam)) > 1
    sel, dem, ms = oracle.best_response(t, 0, full.lam)
    assert np.array_equal(full.min_score, ms) and np.array_equal(full.sel, sel) and np.array_equal(full.demand, dem)
