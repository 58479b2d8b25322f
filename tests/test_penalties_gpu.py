"""The Gamma term of Eq. esp_score on the GPU (esp_set_penalties): switching cost from the current
configuration and the interference penalty above the adaptive threshold, applied as effective values.
Parity with the oracle run on its own penalized values, bit-exact, on every evaluation path."""

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


def penalties(t, rng, gamma0=0.05, alpha=0.4):
    K = np.diff(t.job_off)
    cur = np.array([rng.integers(-1, k) for k in K], np.int32)
    tau = esp.esp_adaptive_threshold(1.1 + 0.2 * rng.random(t.S * t.J), 0.3, 0.9, 0.8, 0.1)
    return dict(gamma0=gamma0, c_cur=cur, alpha=alpha, s_hat=1.0 + 0.6 * rng.random(t.n_opt), tau=tau)


def table(case):
    rng = np.random.default_rng(zlib.crc32(case.encode()))
    if case == "uniform":
        return W.whatif_batch(scenarios=[3, 8], J=700).table
    if case == "ragged":
        return W.random_table(rng, S=3, J=600, R=6, kmin=1, kmax=200)
    if case == "grouped":
        return W.random_table(rng, S=2, J=300, R=6, kmin=1, kmax=400, groups=10, r_global=4)
    if case == "heavy":
        return W.heavy_tail(scenarios=[5], J=4000).table
    raise ValueError(case)


@pytest.mark.parametrize("case,resident", [("uniform", False), ("ragged", False), ("grouped", False),
                                           ("heavy", False), ("uniform", True), ("ragged", True)])
def test_penalties_match_oracle(case, resident):
    t = table(case)
    rng = np.random.default_rng(zlib.crc32((case + "pen").encode()))
    pen = penalties(t, rng)
    s = esp.Solver(t)
    esp.esp_set_penalties(s.ctx, **pen)
    tp = W.OptionTable(**{**t.__dict__, "values": oracle.penalized_values(t, **pen)})
    flags = esp.ESP_FLAG_RESIDENT if resident else 0
    T = 40
    sol = s.solve(0.05, T, flags=flags, traces=True)
    if resident:
        assert s.launches() == 3
    check_solution(tp, sol, list(range(t.S)), 0.05, T, esp.ESP_PRICE_NORMALIZED, esp.ESP_STEP_FIXED)
    # clearing the penalties gives back the unpenalized solve, bit for bit
    esp.esp_set_penalties(s.ctx)
    a = s.solve(0.05, T, flags=flags, traces=True)
    b = esp.Solver(t).solve(0.05, T, flags=flags, traces=True)
    for f in ("lam", "sel", "demand", "lambda_trace", "demand_trace", "selhash_trace"):
        assert np.array_equal(getattr(a, f), getattr(b, f), equal_nan=True), f


def test_large_switching_cost_keeps_current_configurations():
    t = table("ragged")
    rng = np.random.default_rng(4)
    K = np.diff(t.job_off)
    cur = np.array([rng.integers(0, k) for k in K], np.int32)
    s = esp.Solver(t)
    esp.esp_set_penalties(s.ctx, gamma0=1e6, c_cur=cur)
    sol = s.solve(0.05, 30)
    assert np.array_equal(sol.sel.ravel(), cur)


def test_penalties_rejected_and_context_kept():
    t = table("ragged")
    s = esp.Solver(t)
    K = np.diff(t.job_off)
    bad = (K - 1).astype(np.int32)
    bad[7] = K[7]                                   # one past the job's last option
    with pytest.raises(esp.EspError) as e:
        esp.esp_set_penalties(s.ctx, gamma0=0.1, c_cur=bad)
    assert e.value.status == esp.ESP_ERR_INVALID_ARG
    with pytest.raises(esp.EspError):
        esp.esp_set_penalties(s.ctx, gamma0=-1.0)
    ref = esp.Solver(t).solve(0.05, 20)
    got = s.solve(0.05, 20)                          # the loaded values are back
    assert np.array_equal(got.lam, ref.lam) and np.array_equal(got.sel, ref.sel)
