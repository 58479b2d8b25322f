"""The per-round device time trace (esp_params.round_time_trace): for every scenario, the GPU's global
timer when each of its round updates (Eq. price_update) was applied, on every solve path: one launch
per round, the persistent pass, the cluster-resident solve and the grid-resident placement solve.
Entries of rounds a scenario ran are increasing and lie within the solve's device time; entries of
rounds it did not run keep the caller's contents; the rest of the solution is what the solve gives
without the trace."""

import numpy as np
import pytest

from paper_2608_07971_gb300 import esp, workloads as W

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("needs a GPU")
    from paper_2608_07971_gb300 import build
    build.build()
    esp.load_library()


def solve_with_times(s, eta, T, **kw):
    S, J, R, P = s.shape
    prm = s.params(eta, T, **kw)
    tt = np.full((S, T), 7, np.uint64)   # rows of rounds not run must keep this
    prm.round_time_trace = tt.ctypes.data
    res = np.zeros(S, esp.RESULT_DTYPE)
    esp.esp_solve(s.ctx, prm, res)
    lam = np.zeros((S, P))
    esp.esp_get_prices(s.ctx, lam)
    return tt, res, lam


def check_times(tt, res):
    for s in range(tt.shape[0]):
        n = int(res["rounds_run"][s])
        assert n >= 1
        row = tt[s, :n].astype(np.int64)
        assert np.all(np.diff(row) > 0), f"round times of scenario {s} do not increase"
        assert row[-1] - row[0] <= float(res["device_ms"][s]) * 1e6 + 1e6   # within the solve (1 ms slack)
        assert np.all(tt[s, n:] == 7), "rows of rounds not run must be left as they were"


@pytest.mark.parametrize("path", ["per_round", "persistent"])
def test_round_times_streaming(path):
    t = W.whatif_batch(scenarios=[1, 5, 9], J=700).table
    s = esp.Solver()
    esp.esp_debug_set_persistent(s.ctx, 1 if path == "persistent" else 0)
    s.load(t)
    tt, res, lam = solve_with_times(s, 0.05, 30, tol=0.02)
    assert s.launches() == (4 if path == "persistent" else 30 + 3)
    check_times(tt, res)
    plain = s.solve(0.05, 30, tol=0.02)
    assert np.array_equal(plain.lam, lam)
    s.close()


def test_round_times_cluster_resident():
    w = W.tiny_cluster()
    s = esp.Solver(w.table)
    tt, res, lam = solve_with_times(s, w.eta0, 50, flags=esp.ESP_FLAG_RESIDENT)
    assert s.launches() == 3
    check_times(tt, res)
    s.close()


def test_round_times_grid_resident_placement():
    w = W.placement_expanded(J=256)
    s = esp.Solver()
    s.load_placement(w.factors)
    tt, res, lam = solve_with_times(s, w.eta0, 20, flags=esp.ESP_FLAG_RESIDENT)
    assert s.launches() == 4
    check_times(tt, res)
    s.close()
