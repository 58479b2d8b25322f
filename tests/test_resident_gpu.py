"""Parity of the cluster-resident kernel (ESP_FLAG_RESIDENT: all rounds in one launch, each
scenario's table in the shared memory of one thread-block cluster) with the oracle, element by
element, for every cluster size that fits: uniform and CSR layouts, units below and above 2^23,
both price modes and step rules, traces, warm start, the stopping rule, the exact path, non-finite
prices; and bit-identical trajectories with the streaming path.
"""

import zlib

import numpy as np
import pytest

from paper_2608_07971_gb300 import esp, workloads as W
from tests.parity_util import check_solution

pytestmark = pytest.mark.gpu

RES = esp.ESP_FLAG_RESIDENT
SIZES = (1, 2, 4, 8, 16)


@pytest.fixture(scope="module", autouse=True)
def _lib():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("needs a GPU")
    from paper_2608_07971_gb300 import build
    build.build()
    esp.load_library()


def table(case):
    rng = np.random.default_rng(zlib.crc32(case.encode()))
    if case == "tiny":
        return W.tiny_cluster().table
    if case == "whatif3":
        return W.whatif_batch(scenarios=[0, 5, 700]).table
    if case == "ragged":        # CSR layout, K from 1 to 40, ragged slices
        return W.random_table(rng, S=3, J=900, R=6, kmin=1, kmax=40)
    if case == "k5":            # uniform K that is not a power of two
        return W.random_table(rng, S=2, J=1000, R=4, kmin=5, kmax=5)
    if case == "large_units":   # units up to 2^26: int32 storage, converted every round
        return W.random_table(rng, S=2, J=500, R=6, kmin=1, kmax=20, umax=1 << 26)
    if case == "r16":
        return W.random_table(rng, S=2, J=300, R=16, kmin=1, kmax=30)
    if case == "r1":
        return W.random_table(rng, S=2, J=700, R=1, kmin=2, kmax=9)
    if case == "dups":          # many exact duplicates and fp32 ties (dyadic values)
        t = W.random_table(rng, S=2, J=400, R=4, kmin=2, kmax=20, umax=8, dyadic=True)
        for j in range(t.S * t.J):
            a, b = t.job_off[j], t.job_off[j + 1]
            t.units[a + 1:b] = t.units[a]
            t.values[a + 1:b:2] = t.values[a]
        return t
    if case == "few_jobs":      # fewer jobs than CTAs for large clusters: empty slices
        return W.random_table(rng, S=2, J=5, R=3, kmin=1, kmax=60)
    if case == "big_job":       # one job much larger than the rest
        t = W.random_table(rng, S=1, J=64, R=5, kmin=1, kmax=8)
        big = W.random_table(rng, S=1, J=1, R=5, kmin=3000, kmax=3000)
        units = np.concatenate([big.units, t.units])
        values = np.concatenate([big.values, t.values])
        off = np.concatenate([[0], 3000 + t.job_off])
        return W.OptionTable(1, 65, 5, 5, 5, off.astype(np.int64), units, values, None, t.capacity)
    raise ValueError(case)


CASES = ["tiny", "whatif3", "ragged", "k5", "large_units", "r16", "r1", "dups", "few_jobs", "big_job"]


def fitting_sizes(s):
    out = []
    for cs in SIZES:
        try:
            got = esp.esp_debug_resident(s.ctx, cs)
        except esp.EspError:
            continue
        assert got is not None and got[0] == cs and got[1] >= 1
        out.append(cs)
    esp.esp_debug_resident(s.ctx, 0)
    return out


@pytest.mark.parametrize("case", CASES)
def test_resident_every_cluster_size(case):
    t = table(case)
    s = esp.Solver(t)
    sizes = fitting_sizes(s)
    assert sizes, "every test table fits some cluster size"
    T = 40
    for mode, eta in ((esp.ESP_PRICE_NORMALIZED, 0.3), (esp.ESP_PRICE_RAW, 1e-4)):
        ref = s.solve(eta, T, mode=mode, traces=True)                 # streaming path
        assert s.launches() == T + 3
        for cs in sizes:
            esp.esp_debug_resident(s.ctx, cs)
            sol = s.solve(eta, T, mode=mode, flags=RES, traces=True)
            assert s.launches() == 3, "the resident kernel ran"
            check_solution(t, sol, list(range(t.S)), eta, T, mode, esp.ESP_STEP_FIXED)
            for f in ("lam", "sel", "demand", "lambda_trace", "demand_trace", "selhash_trace"):
                assert np.array_equal(getattr(sol, f), getattr(ref, f), equal_nan=True), (cs, f)
        esp.esp_debug_resident(s.ctx, 0)


@pytest.mark.parametrize("mode", [esp.ESP_PRICE_NORMALIZED, esp.ESP_PRICE_RAW])
@pytest.mark.parametrize("step", [esp.ESP_STEP_FIXED, esp.ESP_STEP_INV_SQRT])
def test_resident_tiny_cluster_full(mode, step):
    w = W.tiny_cluster()
    eta = w.eta0 if mode == esp.ESP_PRICE_NORMALIZED else 1e-7
    s = esp.Solver(w.table)
    sol = s.solve(eta, w.rounds, mode=mode, step=step, flags=RES, traces=True)
    assert s.launches() == 3
    check_solution(w.table, sol, [0], eta, w.rounds, mode, step)


def test_resident_cluster_512_full():
    w = W.cluster_512()
    s = esp.Solver(w.table)
    sol = s.solve(w.eta0, w.rounds, flags=RES, traces=True)
    assert s.launches() == 3
    check_solution(w.table, sol, [0], w.eta0, w.rounds, esp.ESP_PRICE_NORMALIZED, esp.ESP_STEP_FIXED)


def test_resident_warm_start_and_tolerance():
    w = W.tiny_cluster()
    t = w.table
    s = esp.Solver(t)
    lam0 = np.abs(np.random.default_rng(1).normal(size=(1, t.P)))
    for cs in fitting_sizes(s):
        esp.esp_debug_resident(s.ctx, cs)
        sol = s.solve(w.eta0, 150, step=esp.ESP_STEP_INV_SQRT, tol=5e-3, lambda0=lam0, flags=RES, traces=True)
        assert s.launches() == 3
        assert sol.result["converged"][0] == 1 and sol.result["rounds_run"][0] < 150   # stops at 74
        check_solution(t, sol, [0], w.eta0, 150, esp.ESP_PRICE_NORMALIZED, esp.ESP_STEP_INV_SQRT, tol=5e-3,
                       lambda0=lam0)


def test_resident_exact_paths():
    rng = np.random.default_rng(9)
    t = W.random_table(rng, S=3, J=100, R=4, kmin=1, kmax=12)
    t.values[: t.n_opt // 3] *= 2.0**120          # beyond the fp32 screen's range
    t.values[t.n_opt // 3: 2 * t.n_opt // 3] *= 2.0**-140   # fp32 subnormal / zero
    s = esp.Solver(t)
    for mode, eta in ((esp.ESP_PRICE_RAW, 1e25), (esp.ESP_PRICE_RAW, 1e-30), (esp.ESP_PRICE_NORMALIZED, 0.2)):
        sol = s.solve(eta, 12, mode=mode, flags=RES, traces=True)
        assert s.launches() == 3
        check_solution(t, sol, [0, 1, 2], eta, 12, mode, esp.ESP_STEP_FIXED)
    w = W.whatif_batch(scenarios=[4], J=512)
    s = esp.Solver(w.table)
    a = s.solve(w.eta0, 30, flags=RES, traces=True)
    b = s.solve(w.eta0, 30, flags=RES | esp.ESP_FLAG_EXACT_ONLY, traces=True)
    for f in ("lam", "sel", "demand", "lambda_trace", "demand_trace", "selhash_trace"):
        assert np.array_equal(getattr(a, f), getattr(b, f), equal_nan=True), f


def test_resident_nonfinite_prices_reported():
    t = W.random_table(np.random.default_rng(2), S=2, J=20, R=2, kmin=1, kmax=3, umax=2**30)
    t.capacity[:] = 1
    s = esp.Solver(t)
    sol = s.solve(1e300, 5, mode=esp.ESP_PRICE_RAW, flags=RES, traces=True)
    assert s.launches() == 3
    assert sol.status == esp.ESP_ERR_OVERFLOW
    check_solution(t, sol, [0, 1], 1e300, 5, esp.ESP_PRICE_RAW, esp.ESP_STEP_FIXED)


def test_resident_zero_rounds():
    t = table("ragged")
    s = esp.Solver(t)
    sol = s.solve(0.1, 0, flags=RES, traces=True)
    assert s.launches() == 3
    check_solution(t, sol, [0, 1, 2], 0.1, 0, esp.ESP_PRICE_NORMALIZED, esp.ESP_STEP_FIXED)


def test_resident_not_taken_where_it_cannot_run():
    """Grouped tables and tables without jobs run the streaming path under ESP_FLAG_RESIDENT."""
    g = W.random_table(np.random.default_rng(8), S=2, J=100, R=6, kmin=1, kmax=30, groups=10, r_global=4)
    s = esp.Solver(g)
    assert esp.esp_debug_resident(s.ctx) is None
    sol = s.solve(0.05, 20, flags=RES, traces=True)
    assert s.launches() == 20 + 3
    check_solution(g, sol, [0, 1], 0.05, 20, esp.ESP_PRICE_NORMALIZED, esp.ESP_STEP_FIXED)
    with pytest.raises(esp.EspError):
        esp.esp_debug_resident(esp.Solver(table("tiny")).ctx, 3)     # not a cluster size


def test_resident_in_graph_with_pass_events():
    """On a non-default stream the resident solve is one CUDA graph; ESP_FLAG_PASS_EVENTS times the
    one resident launch."""
    import torch
    t = W.whatif_batch(scenarios=[0, 1, 2, 3], J=512).table
    st = torch.cuda.Stream()
    s = esp.Solver(t, stream=st.cuda_stream)
    prm = s.params(0.02, 25, flags=RES | esp.ESP_FLAG_PASS_EVENTS)
    for _ in range(3):
        esp.esp_solve_async(s.ctx, prm)
    ms, n = esp.esp_pass_times(s.ctx)
    assert n == 1 and ms > 0.0
    assert s.launches() == 3
    lam = np.zeros((t.S, t.P))
    esp.esp_get_prices(s.ctx, lam)
    ref = esp.Solver(t).solve(0.02, 25)
    assert np.array_equal(lam, ref.lam)


def test_resident_falls_back_to_streaming_when_predicted_slower():
    """A batch of many scenarios needs many waves of clusters: the cost model predicts the resident solve
    slower than streaming, so ESP_FLAG_RESIDENT runs the streaming path (its rounds in one persistent
    launch: 4 launches) with the same results, unless a cluster size is forced. One 2048-job scenario
    keeps the resident solve."""
    w = W.whatif_batch(scenarios=list(range(256)))
    t = w.table
    s = esp.Solver(t)
    assert esp.esp_debug_resident(s.ctx) is not None          # it could run resident ...
    a = s.solve(w.eta0, 20, flags=RES)
    assert s.launches() == 4                                  # ... but streams
    b = s.solve(w.eta0, 20)
    assert np.array_equal(a.lam, b.lam) and np.array_equal(a.sel, b.sel)
    cs, _ = esp.esp_debug_resident(s.ctx)
    esp.esp_debug_resident(s.ctx, cs)                         # a forced size runs resident
    c = s.solve(w.eta0, 20, flags=RES)
    assert s.launches() == 3
    assert np.array_equal(c.lam, b.lam) and np.array_equal(c.sel, b.sel)
    s.close()
    one = esp.Solver(W.cluster_512().table)
    one.solve(0.02, 20, flags=RES)
    assert one.launches() == 3
    one.close()
