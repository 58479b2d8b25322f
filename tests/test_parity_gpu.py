"""Parity of the CUDA path (through the C ABI) with the oracle, element by element.

The bar: selections, integer demands and selection fingerprints bit-exact; the price trajectory
within 1e-12 relative per step (bit-exact is expected: both sides perform the same IEEE operations);
primal and dual objectives within 1e-9 relative (the GPU sums in a fixed tree, the oracle in job
order).
"""

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


# ---------------------------------------------------------------------------------------------
# The benchmark workloads (sizes the oracle finishes in seconds)

@pytest.mark.parametrize("mode", [esp.ESP_PRICE_NORMALIZED, esp.ESP_PRICE_RAW])
@pytest.mark.parametrize("step", [esp.ESP_STEP_FIXED, esp.ESP_STEP_INV_SQRT])
def test_tiny_cluster_full(mode, step):
    w = W.tiny_cluster()
    eta = w.eta0 if mode == esp.ESP_PRICE_NORMALIZED else 1e-7
    s = esp.Solver(w.table)
    sol = s.solve(eta, w.rounds, mode=mode, step=step, traces=True)
    check_solution(w.table, sol, [0], eta, w.rounds, mode, step)


def test_cluster_512_full():
    w = W.cluster_512()
    s = esp.Solver(w.table)
    sol = s.solve(w.eta0, w.rounds, traces=True)
    check_solution(w.table, sol, [0], w.eta0, w.rounds, esp.ESP_PRICE_NORMALIZED, esp.ESP_STEP_FIXED)


def test_whatif_batch_scenarios():
    ids = [0, 1, 2, 77, 512, 1023]
    w = W.whatif_batch(scenarios=ids)
    s = esp.Solver(w.table)
    sol = s.solve(w.eta0, w.rounds, traces=True)
    check_solution(w.table, sol, list(range(len(ids))), w.eta0, w.rounds, esp.ESP_PRICE_NORMALIZED,
                   esp.ESP_STEP_FIXED)


def test_placement_expanded_short():
    w = W.placement_expanded(J=512)
    s = esp.Solver(w.table)
    T = 60
    sol = s.solve(w.eta0, T, traces=True)
    check_solution(w.table, sol, [0], w.eta0, T, esp.ESP_PRICE_NORMALIZED, esp.ESP_STEP_FIXED)


def test_heavy_tail_short():
    w = W.heavy_tail(scenarios=[0, 9], J=8192)
    s = esp.Solver(w.table)
    T = 80
    sol = s.solve(w.eta0, T, traces=True)
    check_solution(w.table, sol, [0, 1], w.eta0, T, esp.ESP_PRICE_NORMALIZED, esp.ESP_STEP_FIXED)


# ---------------------------------------------------------------------------------------------
# Identical prices: esp_evaluate against the oracle's best response (bit-exact selections/demands)

@pytest.mark.parametrize("name", ["tiny_cluster", "cluster_512", "heavy_tail"])
def test_evaluate_at_oracle_prices(name):
    if name == "heavy_tail":
        w = W.heavy_tail(scenarios=[3], J=4096)
    else:
        w = W.make(name)
    t = w.table
    ref = oracle.solve_scenario(t, 0, w.eta0, 40, traces=True)
    s = esp.Solver(t)
    for ti in (0, 5, 17, 39):
        lam = ref.lambda_trace[ti][None, :]
        sel, dem, ms = s.evaluate(lam)
        rsel, rdem, rms = oracle.best_response(t, 0, lam[0], oracle.NORMALIZED)
        assert np.array_equal(sel[0], rsel)
        assert np.array_equal(dem[0], rdem)
        assert np.array_equal(ms[0], rms)     # the minimal reduced cost is the same fp64 chain


# ---------------------------------------------------------------------------------------------
# Ragged, degenerate and extreme tables

@pytest.mark.parametrize("case", ["k1", "ragged", "big_jobs", "tile_edges", "r16", "grouped_many",
                                  "ties", "single_job", "u2", "u32", "u16dups", "u8grouped", "big_dups"])
def test_edge_tables(case):
    rng = np.random.default_rng(zlib.crc32(case.encode()))
    if case == "k1":
        t = W.random_table(rng, S=3, J=1000, R=6, kmin=1, kmax=1)
    elif case == "ragged":
        t = W.random_table(rng, S=4, J=700, R=6, kmin=1, kmax=300)
    elif case == "big_jobs":
        t = W.random_table(rng, S=2, J=9, R=6, kmin=600, kmax=2500)
    elif case == "tile_edges":
        t = W.random_table(rng, S=2, J=300, R=6, kmin=31, kmax=33)
    elif case == "r16":
        t = W.random_table(rng, S=2, J=200, R=16, kmin=1, kmax=70)
    elif case == "grouped_many":
        t = W.random_table(rng, S=2, J=300, R=5, kmin=1, kmax=400, groups=200, r_global=3)
    elif case == "ties":
        t = W.random_table(rng, S=2, J=400, R=4, kmin=2, kmax=20, umax=8, dyadic=True)
        # many exact duplicates
        for j in range(t.S * t.J):
            a, b = t.job_off[j], t.job_off[j + 1]
            t.units[a + 1:b] = t.units[a]
            t.values[a + 1:b:2] = t.values[a]
    elif case == "u2":
        t = W.random_table(rng, S=3, J=333, R=6, kmin=2, kmax=2)
    elif case == "u32":
        t = W.random_table(rng, S=2, J=257, R=4, kmin=32, kmax=32)
    elif case == "u16dups":
        t = W.random_table(rng, S=3, J=500, R=6, kmin=16, kmax=16, umax=6, dyadic=True)
        for j in range(t.S * t.J):
            a = t.job_off[j]
            t.units[a + 8:a + 16] = t.units[a:a + 8]
            t.values[a + 8:a + 16] = t.values[a:a + 8]
    elif case == "big_dups":
        # jobs of 1000 (duplicates marked at load) and 1500 options (too large to mark: resolved
        # by the comparison with the first survivor), most options repeating a few profiles
        t = W.random_table(rng, S=2, J=6, R=6, kmin=1000, kmax=1500, umax=3, dyadic=True)
        for j in range(t.S * t.J):
            a, b = t.job_off[j], t.job_off[j + 1]
            base = np.arange(a, b)
            src = a + (base - a) % 7
            t.units[base] = t.units[src]
            t.values[base] = t.values[src]
    elif case == "u8grouped":
        t = W.random_table(rng, S=2, J=300, R=8, kmin=8, kmax=8, groups=16, r_global=6)
    else:
        t = W.random_table(rng, S=1, J=1, R=3, kmin=5000, kmax=5000)
    for mode, eta in ((esp.ESP_PRICE_NORMALIZED, 0.3), (esp.ESP_PRICE_RAW, 1e-4)):
        s = esp.Solver(t)
        T = 30
        sol = s.solve(eta, T, mode=mode, traces=True)
        check_solution(t, sol, list(range(t.S)), eta, T, mode, esp.ESP_STEP_FIXED)
        exact = s.solve(eta, T, mode=mode, flags=esp.ESP_FLAG_EXACT_ONLY, traces=True)
        assert np.array_equal(exact.sel, sol.sel)
        assert np.array_equal(exact.lambda_trace, sol.lambda_trace)
        assert np.array_equal(exact.demand_trace, sol.demand_trace)


def test_zero_rounds_and_empty_jobs():
    rng = np.random.default_rng(3)
    t = W.random_table(rng, S=2, J=50, R=4, kmin=1, kmax=9)
    s = esp.Solver(t)
    sol = s.solve(0.1, 0, traces=True)
    check_solution(t, sol, [0, 1], 0.1, 0, esp.ESP_PRICE_NORMALIZED, esp.ESP_STEP_FIXED)
    e = W.OptionTable(2, 0, 3, 3, 3, np.zeros(1, np.int64), np.zeros((0, 3), np.int32), np.zeros(0),
                      None, np.full((2, 3), 10, np.int64))
    s2 = esp.Solver(e)
    lam0 = np.full((2, 3), 5.0)
    sol = s2.solve(0.5, 20, mode=esp.ESP_PRICE_RAW, lambda0=lam0, traces=True)
    check_solution(e, sol, [0, 1], 0.5, 20, esp.ESP_PRICE_RAW, esp.ESP_STEP_FIXED, lambda0=lam0)


def test_warm_start_and_tolerance():
    w = W.tiny_cluster()
    t = w.table
    s = esp.Solver(t)
    lam0 = np.abs(np.random.default_rng(1).normal(size=(1, t.P)))
    sol = s.solve(w.eta0, 150, step=esp.ESP_STEP_INV_SQRT, tol=2e-3, lambda0=lam0, traces=True)
    check_solution(t, sol, [0], w.eta0, 150, esp.ESP_PRICE_NORMALIZED, esp.ESP_STEP_INV_SQRT, tol=2e-3,
                   lambda0=lam0)


def test_extreme_magnitudes_take_the_exact_path():
    rng = np.random.default_rng(9)
    t = W.random_table(rng, S=3, J=100, R=4, kmin=1, kmax=12)
    t.values[: t.n_opt // 3] *= 2.0**120          # beyond the fp32 screen's range
    t.values[t.n_opt // 3: 2 * t.n_opt // 3] *= 2.0**-140   # fp32 subnormal / zero
    s = esp.Solver(t)
    for mode, eta in ((esp.ESP_PRICE_RAW, 1e25), (esp.ESP_PRICE_RAW, 1e-30), (esp.ESP_PRICE_NORMALIZED, 0.2)):
        sol = s.solve(eta, 12, mode=mode, traces=True)
        check_solution(t, sol, [0, 1, 2], eta, 12, mode, esp.ESP_STEP_FIXED)


def test_nonfinite_prices_reported():
    t = W.random_table(np.random.default_rng(2), S=2, J=20, R=2, kmin=1, kmax=3, umax=2**30)
    t.capacity[:] = 1
    s = esp.Solver(t)
    sol = s.solve(1e300, 5, mode=esp.ESP_PRICE_RAW, traces=True)
    assert sol.status == esp.ESP_ERR_OVERFLOW
    check_solution(t, sol, [0, 1], 1e300, 5, esp.ESP_PRICE_RAW, esp.ESP_STEP_FIXED)


def test_invalid_tables_rejected():
    rng = np.random.default_rng(4)
    t = W.random_table(rng, S=1, J=10, R=3, kmin=1, kmax=4)
    s = esp.Solver()
    bad = W.OptionTable(**{**t.__dict__, "units": t.units.copy()})
    bad.units[3, 1] = -1
    with pytest.raises(esp.EspError) as e:
        s.load(bad)
    assert e.value.status == esp.ESP_ERR_INVALID_ARG
    bad = W.OptionTable(**{**t.__dict__, "values": t.values.copy()})
    bad.values[2] = np.inf
    with pytest.raises(esp.EspError):
        s.load(bad)
    bad = W.OptionTable(**{**t.__dict__, "capacity": t.capacity.copy()})
    bad.capacity[0, 0] = 0
    with pytest.raises(esp.EspError):
        s.load(bad)
    s.load(t)   # a good table still loads afterwards
    sol = s.solve(0.1, 5)
    assert sol.status == esp.ESP_OK


def test_duplicate_marking_matches_numpy_count():
    """Options equal (units and value bits) to an earlier option of their job are marked at load;
    the count equals an independent per-job count of repeated rows."""
    w = W.whatif_batch(scenarios=[0, 3], J=1024)
    t = w.table
    rows = np.concatenate([t.units.view(np.uint32).reshape(t.n_opt, t.R),
                           t.values.view(np.uint32).reshape(t.n_opt, 2)], axis=1)
    want = 0
    for j in range(t.S * t.J):
        a, b = t.job_off[j], t.job_off[j + 1]
        want += (b - a) - len(np.unique(rows[a:b], axis=0))
    s = esp.Solver(t)
    res, marked = esp.esp_debug_stats(s.ctx)
    assert marked == want and want > 0
    s.solve(w.eta0, 5)
    res, _ = esp.esp_debug_stats(s.ctx)
    assert res <= 0.05 * t.S * t.J * 6          # few exact resolutions once duplicates are marked


@pytest.mark.parametrize("name", ["whatif", "heavy", "grouped"])
def test_fused_update_equals_separate_update_launch(name):
    """The price update done by the last warp of each scenario inside the evaluation pass gives the
    same trajectory as the separate update launch (ESP_FLAG_PER_ROUND_LAUNCH)."""
    if name == "whatif":
        t = W.whatif_batch(scenarios=[2, 9, 40], J=700).table
    elif name == "heavy":
        t = W.heavy_tail(scenarios=[1], J=3000).table
    else:
        t = W.random_table(np.random.default_rng(8), S=3, J=200, R=6, kmin=1, kmax=900, groups=10, r_global=4)
    s = esp.Solver(t)
    a = s.solve(0.05, 40, traces=True)
    b = s.solve(0.05, 40, flags=esp.ESP_FLAG_PER_ROUND_LAUNCH, traces=True)
    for f in ("lam", "sel", "demand", "lambda_trace", "demand_trace", "selhash_trace", "dual_trace"):
        assert np.array_equal(getattr(a, f), getattr(b, f), equal_nan=True), f
    assert s.launches() == 2 * 40 + 3
    s.solve(0.05, 40)
    assert s.launches() == 40 + 3


def test_pass_event_timing_in_graph_and_direct():
    """ESP_FLAG_PASS_EVENTS times every evaluation pass: inside the solve's CUDA graph on a
    non-default stream (latest replay) and with direct launches on the default stream."""
    import torch
    t = W.whatif_batch(scenarios=[0, 1], J=256).table
    st = torch.cuda.Stream()
    s = esp.Solver(t, stream=st.cuda_stream)
    prm = s.params(0.02, 10, flags=esp.ESP_FLAG_PASS_EVENTS)
    for _ in range(3):
        esp.esp_solve_async(s.ctx, prm)
    ms, n = esp.esp_pass_times(s.ctx)
    assert n == 11 and ms > 0.0
    d = esp.Solver(t)            # legacy default stream: direct launches accumulate
    for _ in range(2):
        d.solve(0.02, 10, flags=esp.ESP_FLAG_PASS_EVENTS)
    ms, n = esp.esp_pass_times(d.ctx)
    assert n == 22 and ms > 0.0


@pytest.mark.parametrize("case", ["ragged", "zipf", "k3", "mixed_big", "r5"])
def test_sorted_layout_equals_original_layout(case):
    """General tables are evaluated in a load-time layout sorted into runs of equal-size jobs (with
    never-chosen padding); the trajectory is bit-identical to the original layout's and matches the
    oracle, and outputs come back in the caller's job order."""
    rng = np.random.default_rng(zlib.crc32(case.encode()))
    if case == "ragged":
        t = W.random_table(rng, S=3, J=900, R=6, kmin=1, kmax=140)
    elif case == "zipf":
        t = W.heavy_tail(scenarios=[2, 7], J=3000).table
    elif case == "k3":
        t = W.random_table(rng, S=2, J=600, R=4, kmin=3, kmax=3)
    elif case == "mixed_big":
        t = W.random_table(rng, S=2, J=300, R=8, kmin=1, kmax=400, umax=6, dyadic=True)
    else:
        t = W.random_table(rng, S=2, J=500, R=5, kmin=1, kmax=60)
    a = esp.Solver(t)
    b = esp.Solver()
    esp.esp_debug_set_sorted_layout(b.ctx, False)
    b.load(t)
    for mode, eta in ((esp.ESP_PRICE_NORMALIZED, 0.3), (esp.ESP_PRICE_RAW, 1e-4)):
        sa = a.solve(eta, 40, mode=mode, traces=True)
        sb = b.solve(eta, 40, mode=mode, traces=True)
        for f in ("lam", "sel", "demand", "lambda_trace", "demand_trace", "selhash_trace"):
            assert np.array_equal(getattr(sa, f), getattr(sb, f), equal_nan=True), f
        check_solution(t, sa, list(range(t.S)), eta, 40, mode, esp.ESP_STEP_FIXED)
    ref = oracle.solve_scenario(t, 0, 0.3, 10, traces=True)
    lam = np.tile(ref.lambda_trace[7], (t.S, 1))
    sel, dem, ms = a.evaluate(lam)
    rsel, rdem, rms = oracle.best_response(t, 0, lam[0], oracle.NORMALIZED)
    assert np.array_equal(sel[0], rsel) and np.array_equal(dem[0], rdem) and np.array_equal(ms[0], rms)


@pytest.mark.parametrize("graph", [True, False])
def test_programmatic_dependent_launch_is_transparent(graph):
    """Passes launched as programmatic dependents (forced on for a small table, where the default
    keeps them off) give the oracle's solve, and the same bits as ordinary launches."""
    import torch
    t = W.whatif_batch(scenarios=[1, 4, 6], J=300).table
    stream = torch.cuda.Stream() if graph else None
    s = esp.Solver(t, stream=None if stream is None else stream.cuda_stream)
    T = 30
    sols = {}
    for mode in (1, 0):
        esp.esp_debug_set_pdl(s.ctx, mode)
        sols[mode] = s.solve(0.02, T, traces=True)
    check_solution(t, sols[1], [0, 1, 2], 0.02, T, esp.ESP_PRICE_NORMALIZED, esp.ESP_STEP_FIXED)
    for f in ("lam", "sel", "demand", "lambda_trace", "demand_trace", "selhash_trace", "dual_trace"):
        assert np.array_equal(getattr(sols[1], f), getattr(sols[0], f), equal_nan=True), f
    esp.esp_debug_set_pdl(s.ctx, -1)
    s.close()


@pytest.mark.parametrize("case", ["whatif", "heavy", "ragged256", "k1", "k2", "r4k8", "r5k4", "big_units_k16",
                                  "big_units_ragged"])
def test_interleaved_tiles_equal_separate_arrays(case):
    """The per-warp pass reads each tile's units and values with one bulk copy from a tile-interleaved
    copy of the table (the default wherever every tile allows it) or with two copies from the separate
    arrays: the same bits, round by round, and the oracle's at the end."""
    rng = np.random.default_rng(13)
    if case == "whatif":
        t = W.whatif_batch(scenarios=[3, 40], J=1024).table
    elif case == "heavy":
        t = W.heavy_tail(scenarios=[1, 2], J=3000).table
    elif case == "ragged256":
        t = W.random_table(rng, S=3, J=500, R=6, kmin=1, kmax=256, umax=5000)
    elif case in ("k1", "k2"):
        K = int(case[1])
        t = W.random_table(rng, S=2, J=2000, R=6, kmin=K, kmax=K, umax=5000)
    elif case == "r4k8":
        t = W.random_table(rng, S=2, J=900, R=4, kmin=8, kmax=8, umax=5000)
    elif case == "big_units_k16":     # units up to 2^24: fp32 would not hold them exactly
        t = W.random_table(rng, S=2, J=900, R=6, kmin=16, kmax=16, umax=1 << 24)
    elif case == "big_units_ragged":
        t = W.random_table(rng, S=2, J=700, R=6, kmin=1, kmax=200, umax=1 << 24)
    else:
        t = W.random_table(rng, S=2, J=900, R=5, kmin=4, kmax=4, umax=5000)
    a = esp.Solver(t)
    b = esp.Solver()
    esp.esp_debug_set_interleave(b.ctx, False)
    b.load(t)
    assert esp.esp_debug_pass_kernel(b.ctx) == 0
    c = esp.Solver()
    esp.esp_debug_set_stage_f32(c.ctx, False)
    c.load(t)
    T = 30
    sa = a.solve(0.05, T, traces=True)
    sb = b.solve(0.05, T, traces=True)
    sc = c.solve(0.05, T, traces=True)
    for f in ("lam", "sel", "demand", "lambda_trace", "demand_trace", "selhash_trace"):
        assert np.array_equal(getattr(sa, f), getattr(sb, f), equal_nan=True), f
        assert np.array_equal(getattr(sc, f), getattr(sb, f), equal_nan=True), f
    check_solution(t, sa, list(range(t.S)), 0.05, T, esp.ESP_PRICE_NORMALIZED, esp.ESP_STEP_FIXED)
    if case in ("whatif", "heavy", "ragged256", "r4k8", "r5k4", "big_units_k16", "big_units_ragged"):
        # R = 4, 6, 8 with every unit below 2^23: fp32 units in the interleaved tiles
        f32 = case not in ("r5k4", "big_units_k16", "big_units_ragged")
        assert esp.esp_debug_pass_kernel(a.ctx) == (3 if f32 else 1), "the table should take the interleaved tiles"
        assert esp.esp_debug_pass_kernel(c.ctx) == 1
