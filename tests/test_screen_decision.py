"""The screen's decision rule, restated on the CPU, picks the oracle's best response (no GPU).

Per job, the evaluation kernels take m1 = the smallest screen score q (fp32) and m2 = the second
smallest (counting repeats). When m2 > m1 + 2E (the sum rounded up in fp32) the option holding m1
is the exact argmin; otherwise every option with q <= m1 + 2E is rescored in fp64 and the
lexicographic minimum of (s, local index) is taken. Options that repeat an earlier option of their
job (same units and value) are skipped by the screen: they tie with that option and lose on index.
This test applies the rule to tables full of near-ties (values within 1e-12 of each other,
exact ties between distinct options, repeated options, and one-option jobs), with q restated with
exact fp32 rounding and s taken from the oracle, and requires the oracle's selection for every job
in both price modes."""

from fractions import Fraction

import numpy as np
import pytest

import oracle
from paper_2608_07971_gb300 import workloads as W
from tests.test_screen_bound import bound, ru32, screen


def decide(q, s, dup):
    """Local index chosen by the rule for one job (q fp32 screen scores, s fp64 scores, dup flags)."""
    qq = np.where(dup, np.float32(np.inf), q)
    order = np.lexsort((np.arange(len(qq)), qq))
    m1 = qq[order[0]]
    m2 = qq[order[1]] if len(qq) > 1 else np.float32(np.inf)
    return order[0], m1, m2


def rule(q, s, dup, e2):
    i1, m1, m2 = decide(q, s, dup)
    thr = ru32(Fraction(float(m1)) + Fraction(float(e2)))
    if m2 > thr:
        return int(i1), False
    surv = [k for k in range(len(q)) if not dup[k] and q[k] <= thr]
    return min(surv, key=lambda k: (s[k], k)), True


def near_tie_table(seed, S=2, J=60, R=4):
    rng = np.random.default_rng(seed)
    t = W.random_table(rng, S, J, R, 1, 9, umax=1000, dyadic=True)
    v = t.values.copy()
    u = t.units.copy()
    for j in range(S * J):
        a, b = int(t.job_off[j]), int(t.job_off[j + 1])
        if b - a < 2:
            continue
        kind = j % 4
        if kind == 0:        # a repeat of the first option
            u[b - 1], v[b - 1] = u[a], v[a]
        elif kind == 1:      # values within 1e-12 of each other, same units
            u[a:b] = u[a]
            v[a:b] = v[a] * (1.0 + rng.integers(-3, 4, b - a) * 1e-12)
        elif kind == 2:      # distinct options with equal fp64 scores at zero prices
            v[a + 1] = v[a]
    return W.OptionTable(t.S, t.J, t.R, t.P, t.r_global, t.job_off, u, v, t.group, t.capacity)


@pytest.mark.parametrize("seed", range(4))
@pytest.mark.parametrize("mode", [oracle.RAW, oracle.NORMALIZED])
def test_rule_selects_the_oracle_best_response(seed, mode):
    t = near_tie_table(seed)
    ot = oracle.OracleTable(t)
    rng = np.random.default_rng(50 + seed)
    resolved = decided = 0
    for s in range(t.S):
        a0, b0 = int(t.job_off[s * t.J]), int(t.job_off[(s + 1) * t.J])
        for lam in (np.zeros(t.P), rng.random(t.P) * (1e-3 if mode == oracle.RAW else 0.5),
                    np.full(t.P, 0.0625 if mode == oracle.RAW else 8.0)):
            sel, _, _ = oracle.best_response(ot, s, lam, mode)
            p64 = oracle.effective_prices(ot, s, lam, mode)
            units, values = t.units[a0:b0], t.values[a0:b0]
            E, _ = bound(units, values, p64)
            e2 = np.float32(2.0 * E)
            q_all = screen(units, values, p64)
            for j in range(t.J):
                a, b = int(t.job_off[s * t.J + j]), int(t.job_off[s * t.J + j + 1])
                s_fp64 = [oracle.reduced_cost(ot, o, p64) for o in range(a, b)]
                dup = np.zeros(b - a, bool)
                for k in range(1, b - a):
                    for k2 in range(k):
                        if np.array_equal(t.units[a + k], t.units[a + k2]) and t.values[a + k] == t.values[a + k2]:
                            dup[k] = True
                            break
                k, exact = rule(q_all[a - a0:b - a0], s_fp64, dup, e2)
                assert k == sel[j], (s, j, k, sel[j])
                resolved += exact
                decided += not exact
    assert resolved > 0 and decided > 0
