"""Reloading a context: buffers of the previous table are reused, and the host plan is reused when
the offsets are unchanged. Every solve after a reload must equal the solve of a fresh context."""

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


def fresh(t, eta, T):
    s = esp.Solver(t)
    sol = s.solve(eta, T)
    s.close()
    return sol


def same(a, b):
    for f in ("lam", "sel", "demand"):
        assert np.array_equal(getattr(a, f), getattr(b, f)), f
    for k in ("rounds_run", "primal", "dual", "feasible"):
        assert np.array_equal(a.result[k], b.result[k]), k


def test_reload_same_offsets_new_data_and_new_shapes():
    rng = np.random.default_rng(3)
    a = W.random_table(rng, 3, 40, 4, 1, 9)
    b = W.random_table(rng, 3, 40, 4, 1, 9)                 # other offsets, same shape
    c = W.OptionTable(a.S, a.J, a.R, a.P, a.r_global, a.job_off,   # a's offsets, other data
                      rng.integers(0, 50, a.units.shape).astype(np.int32), rng.random(a.n_opt) * 3.0,
                      None, a.capacity)
    d = W.random_table(rng, 2, 300, 6, 16, 16)              # another shape (uniform)
    s = esp.Solver()
    for t in (a, a, b, a, c, c, d, a, d):
        s.load(t)
        same(s.solve(0.05, 30), fresh(t, 0.05, 30))
    s.close()


def test_reload_rejects_bad_offsets_and_recovers():
    rng = np.random.default_rng(4)
    a = W.random_table(rng, 2, 30, 4, 1, 6)
    bad = W.OptionTable(a.S, a.J, a.R, a.P, a.r_global, a.job_off.copy(), a.units, a.values, None, a.capacity)
    bad.job_off[5] = bad.job_off[4]                          # an empty job
    s = esp.Solver()
    s.load(a)
    with pytest.raises(esp.EspError):
        s.load(bad)
    s.load(a)
    same(s.solve(0.05, 20), fresh(a, 0.05, 20))
    s.close()
