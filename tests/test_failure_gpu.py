"""Failure detection of the evaluation pass, tested without a GPU fault, and allocation failures.

A held stage: the next solve's first round pass announces 16 more bytes on its first warp's first stage
than the stage's copies bring, so that barrier phase never completes (no memory is accessed out of
place). With a host-set wait limit of 20 ms of the GPU's global timer, every wait on it runs out: the
solve reports ESP_ERR_TIMEOUT quickly, the context answers ESP_ERR_STATE from then on, and a new context
on the same device solves bit-exactly, on both layouts of the pass's table. Allocation failures are
injected on the host (esp_debug_fail_alloc): a load that meets one returns ESP_ERR_OOM and leaves no
half-built table behind, and the next load succeeds.
"""

import time

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


@pytest.mark.parametrize("interleave", [True, False], ids=["one_copy_per_tile", "two_copies_per_tile"])
@pytest.mark.parametrize("table", ["uniform", "sorted"])
def test_stage_wait_timeout_reports_and_poisons(interleave, table):
    rng = np.random.default_rng(21)
    if table == "uniform":
        t = W.random_table(rng, S=4, J=2048, R=6, kmin=16, kmax=16, umax=5000)
    else:
        t = W.random_table(rng, S=3, J=1500, R=6, kmin=1, kmax=300, umax=5000)
    s = esp.Solver()
    esp.esp_debug_set_interleave(s.ctx, interleave)
    s.load(t)
    assert esp.esp_debug_pass_kernel(s.ctx) == (3 if interleave else 0)
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
    """Every device allocation of a load, failed one at a time, makes esp_load_options return
    ESP_ERR_OOM without launching on a half-built table; the next load succeeds and solves as a fresh
    context does."""
    rng = np.random.default_rng(31)
    t = W.random_table(rng, S=2, J=300, R=6, kmin=1, kmax=200, umax=5000)
    ref = esp.Solver(t).solve(0.05, 15)
    s = esp.Solver()
    n_fail = 0
    for n in range(80):
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


def test_iac_mma_wait_timeout_reports_and_poisons():
    """The tensor-core IAC kernel's bounded MMA wait: one MMA group left uncommitted (no access out of
    place) makes its warpgroup's wait run out after the host-set limit; the call answers
    ESP_ERR_TIMEOUT, the handle ESP_ERR_STATE from then on, and a new handle predicts exactly as
    before."""
    w = W.iac_batch(S=4)
    rows, pairs = w.rows, w.pairs
    pred = esp.Predictor(w.model)
    ref = pred.predict(rows, pairs, w.c_mem)
    esp.esp_iac_debug_set_wait_limit(pred.h, 20)
    esp.esp_iac_debug_hold_commit(pred.h)
    t0 = time.perf_counter()
    with pytest.raises(esp.EspError) as e:
        pred.predict(rows, pairs, w.c_mem)
    dt = time.perf_counter() - t0
    assert e.value.status == esp.ESP_ERR_TIMEOUT
    assert dt < 10.0, f"the timeout took {dt:.1f} s"
    with pytest.raises(esp.EspError) as e2:
        pred.predict(rows, pairs, w.c_mem)
    assert e2.value.status == esp.ESP_ERR_STATE
    pred.close()
    fresh = esp.Predictor(w.model)
    again = fresh.predict(rows, pairs, w.c_mem)
    fresh.close()
    assert np.array_equal(again, ref)
    fma = esp.Predictor(w.model, path=esp.ESP_IAC_PATH_FMA)
    with pytest.raises(esp.EspError) as e3:
        esp.esp_iac_debug_hold_commit(fma.h)
    assert e3.value.status == esp.ESP_ERR_UNSUPPORTED
    fma.close()
