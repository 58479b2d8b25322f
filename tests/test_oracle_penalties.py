"""Pins of the oracle's Gamma term of Eq. esp_score (switching cost and interference penalty), of the
adaptive threshold of Eq. adaptive_threshold and of the effective capacity of Eq. effective_capacity.
Values are dyadic so every expectation is exact; the expectations are switch prices and selections
derived by hand, not the oracle's formulas retyped."""

import numpy as np

import oracle
from paper_2608_07971_gb300 import workloads as W


def one_job_table(values=(3.0, 2.0), units=(8, 4), cap=10):
    return W.OptionTable(1, 1, 1, 1, 1, np.array([0, 2], np.int64), np.array(units, np.int32).reshape(2, 1),
                         np.array(values), None, np.array([[cap]], np.int64))


def select(table, values, lam):
    t = W.OptionTable(**{**table.__dict__, "values": values})
    sel, dem, ms = oracle.best_response(t, 0, np.array([lam]), oracle.RAW)
    return int(sel[0])


def test_adaptive_threshold_closed_form():
    assert oracle.adaptive_threshold(1.0, 0.25, 0.75, 0.5, 0.5) == 1.125      # 1 + 0.25 * (1.5 - 1)
    assert oracle.adaptive_threshold(1.0, 0.25, 2.0, 0.5, 0.5) == 1.5         # 0.25 * 3 clamped to 0.5
    assert oracle.adaptive_threshold(1.0, 0.25, 0.25, 0.5, 0.5) == 0.875      # below target: not clamped


def test_switching_cost_shifts_switch_price():
    # options (u, v) = (8, 3) and (4, 2), one resource, RAW: s = 8 lam - 3 vs 4 lam - 2.
    # No penalty: option 1 wins for lam > 1/4. Current config 0 with gamma0 = 1/2: option 1 pays
    # 1/2 more and wins only for lam > 3/8. Current config 1: option 0 wins only for lam <= 1/8
    # (tie at 1/8 goes to index 0).
    t = one_job_table()
    plain = oracle.penalized_values(t)
    assert np.array_equal(plain, t.values)
    assert [select(t, plain, x) for x in (0.125, 0.3125, 0.5)] == [0, 1, 1]
    cur0 = oracle.penalized_values(t, gamma0=0.5, c_cur=[0])
    assert [select(t, cur0, x) for x in (0.125, 0.3125, 0.375, 0.40625, 0.5)] == [0, 0, 0, 1, 1]
    cur1 = oracle.penalized_values(t, gamma0=0.5, c_cur=[1])
    assert [select(t, cur1, x) for x in (0.0625, 0.125, 0.15625, 0.3125)] == [0, 0, 1, 1]
    none = oracle.penalized_values(t, gamma0=0.5, c_cur=[-1])
    assert np.array_equal(none, t.values)


def test_interference_penalty_only_above_threshold():
    t = one_job_table()
    tau = np.array([1.25])
    at = oracle.penalized_values(t, alpha=2.0, s_hat=np.array([1.0, 1.25]), tau=tau)
    assert np.array_equal(at, t.values)                   # slowdown at the threshold: no penalty
    above = oracle.penalized_values(t, alpha=2.0, s_hat=np.array([1.0, 1.5]), tau=tau)
    # option 1 loses 2 * 0.25 = 1/2 of value: the switch price moves from 1/4 to 3/8
    assert [select(t, above, x) for x in (0.3125, 0.375, 0.40625)] == [0, 0, 1]
    below = oracle.penalized_values(t, alpha=2.0, s_hat=np.array([0.5, 0.75]), tau=tau)
    assert np.array_equal(below, t.values)                # a speed-up is never a bonus
    both = oracle.penalized_values(t, gamma0=0.5, c_cur=[0], alpha=2.0, s_hat=np.array([1.0, 1.5]), tau=tau)
    # switching (1/2) and interference (1/2) add: option 1 needs 4 lam > 2, lam > 1/2
    assert [select(t, both, x) for x in (0.5, 0.53125)] == [0, 1]


def test_large_switching_cost_keeps_current_configuration():
    rng = np.random.default_rng(17)
    for seed in range(4):
        t = W.random_table(np.random.default_rng(seed), S=1, J=6, R=3, kmin=1, kmax=4, dyadic=True)
        K = np.diff(t.job_off)
        cur = np.array([rng.integers(0, k) for k in K], np.int32)
        v = oracle.penalized_values(t, gamma0=1e6, c_cur=cur)
        tp = W.OptionTable(**{**t.__dict__, "values": v})
        for _ in range(5):
            lam = rng.random(t.P) * 0.05
            sel, _, _ = oracle.best_response(tp, 0, lam, oracle.RAW)
            assert np.array_equal(sel, cur)
        ref = oracle.solve_scenario(tp, 0, 1e-3, 20, mode=oracle.RAW)
        assert np.array_equal(ref.sel, cur)


def test_effective_capacity_hand_example():
    cap = np.array([100, 50], np.int64)
    q_off = np.array([0, 2, 3], np.int64)
    # minimum footprints (7, 5) and (3, 3): each column's minimum of the first job comes from its
    # second option, so every column is reduced separately
    q_units = np.array([[10, 9], [7, 5], [3, 3]], np.int32)
    assert np.array_equal(oracle.effective_capacity(cap, q_off, q_units, 0.5), [95, 46])
    assert np.array_equal(oracle.effective_capacity(cap, q_off, q_units, 0.0), [100, 50])
    assert np.array_equal(oracle.effective_capacity(cap, q_off, q_units, 20.0), [1, 1])   # kept >= 1
    assert np.array_equal(oracle.effective_capacity(cap, np.array([0], np.int64), np.zeros((0, 2), np.int32), 1.0),
                          [100, 50])
