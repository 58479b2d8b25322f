"""The streaming evaluation pass (k_stream: a producer warp per CTA filling a ring of stages by bulk
copies, consumer warps evaluating them) against the oracle and against the per-warp pass.

Parity bar as everywhere (Sec. 3.2.2-3.2.3): selections, integer demands and selection fingerprints
bit-exact; prices within 1e-12 relative per step (bit-exact expected); objectives within 1e-9. The
tables cover every path of the streaming pass: uniform jobs of 1, 2, 4, 8, 16 and 32 options (R = 4,
5, 6, 8), and ragged jobs of 1 to 256 options through the sorted layout (runs of 4m options with one or
two groups of four options per lane, runs of one and two options), several blocks per CTA and
scenarios that straddle blocks and CTAs. Failure detection: a stage whose barrier phase never
completes (more bytes announced than copied; no memory is accessed out of place) makes the solve
return ESP_ERR_TIMEOUT within the host-set wait limit, poisons the context, and leaves the device
usable. Allocation failures injected on the host make a load return ESP_ERR_OOM cleanly.
"""

import time

import numpy as np
import pytest

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


def ragged(seed, S, J, R, kmax, dups=True):
    rng = np.random.default_rng(seed)
    t = W.random_table(rng, S=S, J=J, R=R, kmin=1, kmax=kmax, umax=5000)
    if dups:   # exact duplicates inside jobs (marked at load) and near ties
        for j in range(0, S * J, 7):
            a, b = t.job_off[j], t.job_off[j + 1]
            if b - a >= 3:
                t.units[a + 2] = t.units[a]
                t.values[a + 2] = t.values[a]
    return t


def streaming(t=None, stream=True):
    """A context whose loads take the streaming pass (stream=True) or the per-warp pass."""
    s = esp.Solver()
    esp.esp_debug_set_stream_pass(s.ctx, stream)
    if t is not None:
        s.load(t)
    return s


def uniform(seed, S, J, R, K):
    rng = np.random.default_rng(seed)
    return W.random_table(rng, S=S, J=J, R=R, kmin=K, kmax=K, umax=5000)


TABLES = [
    ("uniform_k16_r6", lambda: uniform(1, 5, 700, 6, 16)),
    ("uniform_k32_r4", lambda: uniform(2, 3, 900, 4, 32)),
    ("uniform_k8_r8", lambda: uniform(3, 4, 1000, 8, 8)),
    ("uniform_k4_r5", lambda: uniform(4, 3, 1200, 5, 4)),
    ("uniform_k2_r6", lambda: uniform(5, 3, 1500, 6, 2)),
    ("uniform_k1_r6", lambda: uniform(6, 2, 3000, 6, 1)),
    ("ragged_256_r6", lambda: ragged(7, 4, 600, 6, 256)),
    ("ragged_40_r4", lambda: ragged(8, 6, 800, 4, 40)),
    ("ragged_140_r8", lambda: ragged(9, 3, 500, 8, 140)),
    ("heavy_tail_small", lambda: W.heavy_tail(scenarios=[0, 3], J=2000).table),
    ("whatif_small", lambda: W.whatif_batch(scenarios=[4, 9, 100], J=1024).table),
]


@pytest.mark.parametrize("name,make", TABLES, ids=[n for n, _ in TABLES])
@pytest.mark.parametrize("mode", [esp.ESP_PRICE_NORMALIZED, esp.ESP_PRICE_RAW])
def test_stream_pass_matches_oracle(name, make, mode):
    t = make()
    eta = 0.05 if mode == esp.ESP_PRICE_NORMALIZED else 2e-9
    T = 25
    s = streaming(t)
    assert esp.esp_debug_pass_kernel(s.ctx) == 1, "the table should take the streaming pass"
    sol = s.solve(eta, T, mode=mode, traces=True)
    check_solution(t, sol, list(range(t.S)), eta, T, mode, esp.ESP_STEP_FIXED)
    s.close()


@pytest.mark.parametrize("name,make", TABLES[:3] + TABLES[6:], ids=[n for n, _ in TABLES[:3] + TABLES[6:]])
def test_stream_pass_equals_per_warp_pass(name, make):
    """The streaming and per-warp passes give the same bits, round by round, without traces (the plain
    round-pass kernels) and with the final pass's outputs."""
    t = make()
    T = 40
    a = streaming(t)
    b = streaming(t, stream=False)
    assert esp.esp_debug_pass_kernel(a.ctx) == 1 and esp.esp_debug_pass_kernel(b.ctx) in (0, 3)
    for flags in (0, esp.ESP_FLAG_EXACT_ONLY):
        sa = a.solve(0.03, T, flags=flags)
        sb = b.solve(0.03, T, flags=flags)
        assert np.array_equal(sa.lam, sb.lam)
        assert np.array_equal(sa.sel, sb.sel)
        assert np.array_equal(sa.demand, sb.demand)
        for k in ("primal", "dual", "rounds_run", "feasible"):
            assert np.array_equal(sa.result[k], sb.result[k]), k
        assert np.all(sa.result["device_ms"] > 0)
    rng = np.random.default_rng(3)
    lam = rng.exponential(20.0, size=(t.S, t.P))
    ea, eb = a.evaluate(lam), b.evaluate(lam)
    for x, y in zip(ea, eb):
        assert np.array_equal(x, y)
    a.close()
    b.close()


def test_stream_pass_tolerance_stop_and_warm_start():
    t = ragged(11, 5, 400, 6, 200)
    T = 60
    s = streaming(t)
    sol = s.solve(0.05, T, tol=1e-3, traces=True)
    check_solution(t, sol, list(range(t.S)), 0.05, T, esp.ESP_PRICE_NORMALIZED, esp.ESP_STEP_FIXED, tol=1e-3)
    lam0 = np.random.default_rng(2).exponential(1.0, size=(t.S, t.P))
    sol = s.solve(0.05, 20, step=esp.ESP_STEP_INV_SQRT, lambda0=lam0, traces=True)
    check_solution(t, sol, list(range(t.S)), 0.05, 20, esp.ESP_PRICE_NORMALIZED, esp.ESP_STEP_INV_SQRT,
                   lambda0=lam0)
    s.close()


@pytest.mark.parametrize("stream", [True, False], ids=["streaming", "per_warp"])
def test_stage_wait_timeout_reports_and_poisons(stream):
    """A held stage: its barrier phase is announced 16 bytes more than its copies bring, so every wait
    on it runs out (after the host-set limit of 20 ms of the GPU's timer); the solve reports
    ESP_ERR_TIMEOUT, the context answers ESP_ERR_STATE, and a new context on the device solves
    bit-exactly."""
    t = uniform(21, 4, 2048, 6, 16)
    s = streaming(t, stream)
    assert esp.esp_debug_pass_kernel(s.ctx) in ((1,) if stream else (0, 3))
    ref = s.solve(0.05, 10)
    esp.esp_debug_set_wait_limit(s.ctx, 20)
    esp.esp_debug_hold_stage(s.ctx)
    t0 = time.perf_counter()
    with pytest.raises(esp.EspError) as e:
        s.solve(0.05, 10)
    dt = time.perf_counter() - t0
    assert e.value.status == esp.ESP_ERR_TIMEOUT
    assert dt < 10.0, f"the timeout took {dt:.1f} s"
    with pytest.raises(esp.EspError) as e2:
        s.solve(0.05, 10)
    assert e2.value.status == esp.ESP_ERR_STATE
    s.close()
    fresh = esp.Solver(t)
    again = fresh.solve(0.05, 10)
    assert np.array_equal(again.lam, ref.lam) and np.array_equal(again.sel, ref.sel)
    fresh.close()


def test_allocation_failure_is_reported_and_recoverable():
    """Every device allocation of a load, failed one at a time on the host, makes esp_load_options
    return ESP_ERR_OOM without launching on a half-built table; the next load succeeds and solves as a
    fresh context does."""
    t = ragged(31, 2, 300, 6, 120)
    ref = esp.Solver(t).solve(0.05, 15)
    s = esp.Solver()
    n_fail = 0
    for n in range(60):
        esp.esp_debug_fail_alloc(s.ctx, n)
        try:
            s.load(t)
        except esp.EspError as e:
            assert e.status == esp.ESP_ERR_OOM, e
            n_fail += 1
            assert esp.load_library().esp_solve(s.ctx, s.params(0.05, 15), None) == esp.ESP_ERR_NOT_LOADED
            continue
        break
    assert n_fail >= 10, "a load makes more than ten allocations"
    esp.esp_debug_fail_alloc(s.ctx, -1)
    s.load(t)
    sol = s.solve(0.05, 15)
    assert np.array_equal(sol.lam, ref.lam) and np.array_equal(sol.sel, ref.sel)
    s.close()
