"""Parity at the full benchmark sizes, in the launch configuration bench.py times (a non-default stream,
one CUDA graph per solve, the price update fused into the evaluation pass, no traces).

The two batched workloads are compared with the oracle scenario by scenario, every scenario of the
batch (1024 what-if scenarios, 16 heavy-tailed ones): the final selections, demands and prices of the
timed launch configuration bit-exact / 1e-12, objectives 1e-9, and, from a second solve that records
the trajectories, the prices of every round within 1e-12 and the demand of every round bit-exact (the
oracle runs in a pool of spawned processes, started before the GPU solves, tests/oracle_batch.py).
The other workloads are compared on their scenario. Every scenario is also checked against properties
that hold at any size: prices finite and non-negative, selections inside each job, the final demand
equal to the units of the selected options, the primal equal to their values, feasibility consistent.
"""

import numpy as np
import pytest

import oracle
from paper_2608_07971_gb300 import esp, workloads as W

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def torch():
    t = pytest.importorskip("torch")
    if not t.cuda.is_available():
        pytest.skip("needs a GPU")
    from paper_2608_07971_gb300 import build
    build.build()
    esp.load_library()
    return t


def solve_like_bench(torch, w, T):
    t = w.table
    stream = torch.cuda.Stream()
    s = esp.Solver(t, stream=stream.cuda_stream)
    prm = s.params(w.eta0, T, mode=w.mode, step=w.step)
    esp.esp_solve_async(s.ctx, prm)
    res = np.zeros(t.S, esp.RESULT_DTYPE)
    esp.esp_get_result(s.ctx, res)
    lam = np.zeros((t.S, t.P))
    sel = np.zeros((t.S, t.J), np.int32)
    dem = np.zeros((t.S, t.P), np.int64)
    esp.esp_get_prices(s.ctx, lam)
    esp.esp_get_selection(s.ctx, sel)
    esp.esp_get_demand(s.ctx, dem)
    # the rounds in one persistent launch where the table takes it, else one launch per round
    assert s.launches() == (4 if esp.esp_debug_persistent(s.ctx) else T + 3)
    s.close()
    return lam, sel, dem, res


def check_properties(t, lam, sel, dem, res, T):
    K = np.diff(t.job_off).reshape(t.S, t.J)
    assert np.all(np.isfinite(lam)) and np.all(lam >= 0.0)
    assert np.all(sel >= 0) and np.all(sel < K)
    assert np.all(res["rounds_run"] == T) and np.all(res["status"] == 0)
    picked = t.job_off[:-1] + sel.ravel()
    u = t.units[picked].astype(np.int64).reshape(t.S, t.J, t.R)
    if t.group is None:
        assert np.array_equal(dem, u.sum(axis=1))
    v = t.values[picked].reshape(t.S, t.J)
    primal = v.sum(axis=1)
    assert np.allclose(res["primal"], primal, rtol=1e-9, atol=0)
    assert np.array_equal(res["feasible"].astype(bool), np.all(dem <= t.capacity, axis=1))


def check_against_oracle(t, w, T, lam, sel, dem, res, scenarios):
    ot = oracle.OracleTable(t)
    for s in scenarios:
        ref = oracle.solve_scenario(ot, s, w.eta0, T, mode=w.mode, step=w.step)
        assert np.array_equal(sel[s], ref.sel), f"selection differs in scenario {s}"
        assert np.array_equal(dem[s], ref.demand), f"demand differs in scenario {s}"
        d = np.abs(lam[s] - ref.lam)
        assert np.all(d <= 1e-12 * np.maximum(np.abs(ref.lam), 1e-300)), f"prices differ in scenario {s}"
        assert res["rounds_run"][s] == ref.rounds_run
        assert abs(res["primal"][s] - ref.primal) <= 1e-9 * max(1.0, abs(ref.primal))
        assert abs(res["dual"][s] - ref.dual) <= 1e-9 * max(1.0, abs(ref.dual))


def check_every_scenario(torch, name):
    """Every scenario of a batched workload against the oracle (started first, in the background)."""
    from tests.oracle_batch import Batch
    w0 = W.make(name, scenarios=[0])
    T = w0.rounds
    S = {"whatif_batch": 1024, "heavy_tail": 16}[name]
    batch = Batch(name, range(S), T)
    w = W.make(name)
    t = w.table
    lam, sel, dem, res = solve_like_bench(torch, w, T)
    check_properties(t, lam, sel, dem, res, T)
    s = esp.Solver(t)
    tr = s.solve(w.eta0, T, mode=w.mode, step=w.step, traces="prices")
    s.close()
    assert np.array_equal(tr.lam, lam) and np.array_equal(tr.sel, sel) and np.array_equal(tr.demand, dem)
    refs = batch.result()
    for i in range(S):
        ref = refs[i]
        assert np.array_equal(sel[i], ref["sel"]), f"selection differs in scenario {i}"
        assert np.array_equal(dem[i], ref["demand"]), f"demand differs in scenario {i}"
        d = np.abs(lam[i] - ref["lam"])
        assert np.all(d <= 1e-12 * np.maximum(np.abs(ref["lam"]), 1e-300)), f"prices differ in scenario {i}"
        assert res["rounds_run"][i] == int(ref["rounds_run"]) == T
        assert res["feasible"][i] == int(ref["feasible"])
        assert abs(res["primal"][i] - float(ref["primal"])) <= 1e-9 * max(1.0, abs(float(ref["primal"])))
        assert abs(res["dual"][i] - float(ref["dual"])) <= 1e-9 * max(1.0, abs(float(ref["dual"])))
        lt = ref["lambda_trace"]
        d = np.abs(tr.lambda_trace[i] - lt)
        assert np.all(d <= 1e-12 * np.maximum(np.abs(lt), 1e-300)), f"price trajectory differs in scenario {i}"
        assert np.array_equal(tr.demand_trace[i], ref["demand_trace"]), f"demand trajectory differs in {i}"


def test_whatif_batch_every_scenario(torch):
    check_every_scenario(torch, "whatif_batch")


def test_heavy_tail_every_scenario(torch):
    check_every_scenario(torch, "heavy_tail")


def test_placement_expanded_full(torch):
    w = W.placement_expanded()
    T = w.rounds
    lam, sel, dem, res = solve_like_bench(torch, w, T)
    check_properties(w.table, lam, sel, dem, res, T)
    check_against_oracle(w.table, w, T, lam, sel, dem, res, [0])


def test_cluster_and_tiny_full(torch):
    for w in (W.tiny_cluster(), W.cluster_512()):
        T = w.rounds
        lam, sel, dem, res = solve_like_bench(torch, w, T)
        check_properties(w.table, lam, sel, dem, res, T)
        check_against_oracle(w.table, w, T, lam, sel, dem, res, [0])


def test_placement_factored_full(torch):
    """The benchmark's placement workload loaded in factored form, full size, against the oracle."""
    w = W.placement_expanded()
    T = w.rounds
    stream = torch.cuda.Stream()
    s = esp.Solver(stream=stream.cuda_stream)
    s.load_placement(w.factors)
    prm = s.params(w.eta0, T, mode=w.mode, step=w.step)
    esp.esp_solve_async(s.ctx, prm)
    t = w.table
    res = np.zeros(t.S, esp.RESULT_DTYPE)
    esp.esp_get_result(s.ctx, res)
    lam = np.zeros((t.S, t.P))
    sel = np.zeros((t.S, t.J), np.int32)
    dem = np.zeros((t.S, t.P), np.int64)
    esp.esp_get_prices(s.ctx, lam)
    esp.esp_get_selection(s.ctx, sel)
    esp.esp_get_demand(s.ctx, dem)
    s.close()
    check_against_oracle(t, w, T, lam, sel, dem, res, [0])
