"""The evaluation pass on every table shape it specializes for, against the oracle.

Parity bar as everywhere (Sec. 3.2.2-3.2.3): selections, integer demands and selection fingerprints
bit-exact; prices within 1e-12 relative per step (bit-exact expected); objectives within 1e-9. The
tables cover the uniform kernel with jobs of 1, 2, 4, 8, 16 and 32 options (R = 4, 5, 6, 8), the
runs-only kernel on sorted layouts of ragged jobs of 1 to 256 options (runs of 4m options, runs of one
and two options, chunked jobs above 128 options), with exact duplicates and near ties, in both price
units, a tolerance stop and a warm start with the 1/sqrt(t) step.
"""

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
def test_pass_matches_oracle(name, make, mode):
    t = make()
    eta = 0.05 if mode == esp.ESP_PRICE_NORMALIZED else 2e-9
    T = 25
    s = esp.Solver(t)
    sol = s.solve(eta, T, mode=mode, traces=True)
    check_solution(t, sol, list(range(t.S)), eta, T, mode, esp.ESP_STEP_FIXED)
    s.close()


def test_tolerance_stop_and_warm_start():
    t = ragged(11, 5, 400, 6, 200)
    T = 60
    s = esp.Solver(t)
    sol = s.solve(0.05, T, tol=1e-3, traces=True)
    check_solution(t, sol, list(range(t.S)), 0.05, T, esp.ESP_PRICE_NORMALIZED, esp.ESP_STEP_FIXED, tol=1e-3)
    lam0 = np.random.default_rng(2).exponential(1.0, size=(t.S, t.P))
    sol = s.solve(0.05, 20, step=esp.ESP_STEP_INV_SQRT, lambda0=lam0, traces=True)
    check_solution(t, sol, list(range(t.S)), 0.05, 20, esp.ESP_PRICE_NORMALIZED, esp.ESP_STEP_INV_SQRT,
                   lambda0=lam0)
    assert np.all(sol.result["device_ms"] > 0)
    s.close()
