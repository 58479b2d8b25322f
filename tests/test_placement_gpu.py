"""Factored placement tables (esp_load_placement): the solve computed from configurations x nodes
without storing the expanded options equals the oracle's solve of the expanded table (and the
streaming solve of that table) bit for bit."""

import time
import zlib

import numpy as np
import pytest

import oracle
from paper_2608_07971_gb300 import esp, workloads as W
from tests.parity_util import check_solution

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("needs a GPU")
    from paper_2608_07971_gb300 import build
    build.build()
    esp.load_library()


def expand(f):
    """The expanded table the factors stand for (include/esp.h's definition, restated)."""
    nj = f.S * f.J
    pen = (f.sens[:, None] * f.D[f.job_type][:, f.node_type]).astype(np.float32)
    values = f.cfg_values[:, :, None] - pen[:, None, :].astype(np.float64)
    units = np.broadcast_to(f.cfg_units[:, :, None, :], (nj, f.KC, f.N, f.R))
    group = np.broadcast_to(np.arange(f.N, dtype=np.uint16)[None, None, :], (nj, f.KC, f.N))
    P = f.r_global + (f.R - f.r_global) * f.N
    off = np.arange(nj + 1, dtype=np.int64) * (f.KC * f.N)
    return W.OptionTable(f.S, f.J, f.R, P, f.r_global, off, np.ascontiguousarray(units.reshape(-1, f.R)),
                         np.ascontiguousarray(values.reshape(-1)), np.ascontiguousarray(group.reshape(-1)),
                         f.capacity)


def random_factors(seed, S=2, J=150, KC=7, N=40, R=5, rg=3, NT=10, dups=True):
    rng = np.random.default_rng(seed)
    nj = S * J
    cu = rng.integers(0, 60, (nj, KC, R)).astype(np.int32)
    cv = np.exp(rng.standard_normal((nj, KC)))
    if dups:                                   # some configurations repeat an earlier one
        cu[::3, KC - 1] = cu[::3, 0]
        cv[::3, KC - 1] = cv[::3, 0]
    P = rg + (R - rg) * N
    cap = np.maximum(1, (0.4 * J * 30 * np.ones((S, P)))).astype(np.int64)
    cap[:, rg:] //= N
    return W.PlacementFactors(S, J, KC, N, R, rg, cu, cv, rng.random(nj).astype(np.float32),
                              rng.integers(0, NT, nj).astype(np.int32), rng.integers(0, NT, N).astype(np.int32),
                              rng.random((NT, NT)).astype(np.float32), cap)


@pytest.mark.parametrize("case", ["bench_shape", "generic"])
@pytest.mark.parametrize("mode", [esp.ESP_PRICE_NORMALIZED, esp.ESP_PRICE_RAW])
def test_factored_placement_matches_oracle(case, mode):
    if case == "bench_shape":
        f = W.placement_expanded(scenarios=[0, 3], J=256).factors
    else:
        f = random_factors(zlib.crc32(b"generic"))
    t = expand(f)
    eta = 0.05 if mode == esp.ESP_PRICE_NORMALIZED else 2e-5
    T = 40
    s = esp.Solver()
    s.load_placement(f)
    sol = s.solve(eta, T, mode=mode, traces=True)
    assert s.launches() == T + 3
    check_solution(t, sol, list(range(t.S)), eta, T, mode, esp.ESP_STEP_FIXED)
    ref = esp.Solver(t).solve(eta, T, mode=mode, traces=True)       # the expanded table, streamed
    for fld in ("lam", "sel", "demand", "lambda_trace", "demand_trace", "selhash_trace"):
        assert np.array_equal(getattr(sol, fld), getattr(ref, fld), equal_nan=True), fld
    ex = s.solve(eta, T, mode=mode, flags=esp.ESP_FLAG_EXACT_ONLY, traces=True)
    assert np.array_equal(ex.lambda_trace, sol.lambda_trace) and np.array_equal(ex.sel, sol.sel)
    sep = s.solve(eta, T, mode=mode, flags=esp.ESP_FLAG_PER_ROUND_LAUNCH, traces=True)
    assert np.array_equal(sep.lambda_trace, sol.lambda_trace)


def test_factored_placement_evaluate_at_oracle_prices():
    f = random_factors(7, S=1, J=300)
    t = expand(f)
    s = esp.Solver()
    s.load_placement(f)
    ref = oracle.solve_scenario(t, 0, 0.05, 25, traces=True)
    for ti in (0, 9, 24):
        lam = ref.lambda_trace[ti][None, :]
        sel, dem, ms = s.evaluate(lam)
        rsel, rdem, rms = oracle.best_response(t, 0, lam[0], oracle.NORMALIZED)
        assert np.array_equal(sel[0], rsel) and np.array_equal(dem[0], rdem) and np.array_equal(ms[0], rms)


def test_factored_placement_rejects_bad_input():
    f = random_factors(3, S=1, J=20)
    bad = W.PlacementFactors(**{**f.__dict__, "job_type": f.job_type.copy()})
    bad.job_type[4] = 99
    s = esp.Solver()
    with pytest.raises(esp.EspError):
        s.load_placement(bad)
    s.load_placement(f)
    with pytest.raises(esp.EspError) as e:
        esp.esp_set_penalties(s.ctx, gamma0=0.1)
    assert e.value.status == esp.ESP_ERR_UNSUPPORTED


def same_solution(a, b, fields=("lam", "sel", "demand", "lambda_trace", "demand_trace")):
    for fld in fields:
        x, y = getattr(a, fld), getattr(b, fld)
        if x is None and y is None:
            continue
        assert np.array_equal(x, y, equal_nan=True), fld
    for k in ("rounds_run", "converged", "feasible", "status", "primal", "dual"):
        assert np.array_equal(a.result[k], b.result[k]), k


@pytest.mark.parametrize("case", ["bench_shape", "generic", "one_job_per_warp"])
@pytest.mark.parametrize("mode", [esp.ESP_PRICE_NORMALIZED, esp.ESP_PRICE_RAW])
def test_grid_resident_placement_equals_per_round_launches(case, mode):
    """ESP_FLAG_RESIDENT on a placement table: every round in one cooperative launch with a grid
    barrier per round; every CTA applies Eq. price_update to its own copy of the prices. The result
    equals the per-round launches bit for bit (and so the expanded table's streaming solve)."""
    if case == "bench_shape":
        f = W.placement_expanded(scenarios=[0, 3], J=256).factors
    elif case == "generic":
        f = random_factors(zlib.crc32(b"resident"), S=3, J=97)
    else:
        f = random_factors(5, S=1, J=7, KC=3, N=9)
    eta = 0.05 if mode == esp.ESP_PRICE_NORMALIZED else 2e-5
    T = 37
    s = esp.Solver()
    s.load_placement(f)
    ref = s.solve(eta, T, mode=mode, traces="prices")
    assert s.launches() == T + 3
    res = s.solve(eta, T, mode=mode, flags=esp.ESP_FLAG_RESIDENT, traces="prices")
    assert s.launches() == 4
    same_solution(res, ref)
    again = s.solve(eta, T, mode=mode, flags=esp.ESP_FLAG_RESIDENT)      # buffers reused, graph replayed
    same_solution(again, ref, fields=("lam", "sel", "demand"))
    full = s.solve(eta, T, mode=mode, flags=esp.ESP_FLAG_RESIDENT, traces=True)   # hash / dual traces:
    assert s.launches() == T + 3                                                    # per-round launches
    same_solution(full, ref)


def test_grid_resident_placement_stops_like_per_round_launches():
    f = random_factors(11, S=2, J=120)
    s = esp.Solver()
    s.load_placement(f)
    for tol, T in ((5e-2, 300), (2e-2, 300), (0.0, 0), (0.0, 1)):
        ref = s.solve(0.05, T, tol=tol, traces="prices")
        res = s.solve(0.05, T, tol=tol, flags=esp.ESP_FLAG_RESIDENT, traces="prices")
        same_solution(res, ref)
        if tol > 0:
            assert (res.result["converged"] == 1).any() and (res.result["rounds_run"] < T).any()  # oracle: 170, 134 at 5e-2; 293 and no stop at 2e-2


def test_grid_resident_placement_full_size():
    """The benchmark placement table (4096 jobs x 12 configurations x 64 nodes, 400 rounds)."""
    w = W.placement_expanded()
    s = esp.Solver()
    s.load_placement(w.factors)
    ref = s.solve(w.eta0, w.rounds)
    res = s.solve(w.eta0, w.rounds, flags=esp.ESP_FLAG_RESIDENT)
    assert s.launches() == 4
    same_solution(res, ref, fields=("lam", "sel", "demand"))


def test_grid_barrier_timeout_is_reported_and_poisons_the_context():
    """Failure detection of the grid-resident solve without a GPU fault: with the barrier held (its
    arrival counter far short of every target, a count that nothing completes) each CTA's bounded
    wait gives up, at its 4 s limit or on the abort word of the first CTA that gave up; the solve
    returns ESP_ERR_TIMEOUT, the context answers ESP_ERR_STATE, and a new context on the same device
    solves correctly."""
    f = random_factors(zlib.crc32(b"resident"), S=3, J=97)    # 291 jobs: 19 CTAs share the barrier
    s = esp.Solver()
    s.load_placement(f)
    ref = s.solve(0.05, 9)
    esp.esp_debug_hold_barrier(s.ctx)
    t0 = time.monotonic()
    with pytest.raises(esp.EspError) as e:
        s.solve(0.05, 9, flags=esp.ESP_FLAG_RESIDENT)
    assert e.value.status == esp.ESP_ERR_TIMEOUT
    assert time.monotonic() - t0 < 60
    with pytest.raises(esp.EspError) as e:
        s.solve(0.05, 9)
    assert e.value.status == esp.ESP_ERR_STATE
    s.close()
    s2 = esp.Solver()
    with pytest.raises(esp.EspError) as e:
        esp.esp_debug_hold_barrier(s2.ctx)                       # nothing loaded
    assert e.value.status == esp.ESP_ERR_UNSUPPORTED
    s2.load_placement(f)
    same_solution(s2.solve(0.05, 9, flags=esp.ESP_FLAG_RESIDENT), ref, fields=("lam", "sel", "demand"))
    s2.close()
