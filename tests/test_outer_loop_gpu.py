"""The outer ESP-IAC loop of Alg. 1 on the GPU: warm-started tatonnement, the IAC predictor's
slowdowns for every option against its co-located partner's current configuration (Sec. 3.3,
Eq. dnn_pred), the adaptive thresholds (Eq. adaptive_threshold) and the Gamma term of Eq.
esp_score set for the next round (esp_set_penalties). Every outer round is compared with the oracle
running the same loop on the same predicted slowdowns: selections and prices bit-exact. The
predictions themselves are checked against the IAC oracle within the tensor path's bound."""

import numpy as np
import pytest

import oracle
from oracle import iac_oracle
from paper_2608_07971_gb300 import esp, workloads as W
from tests import test_iac_gpu as iac_t

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("needs a GPU")
    from paper_2608_07971_gb300 import build
    build.build()
    esp.load_library()


def colocation_pairs(S, J, K, sel):
    """Option (s, j, k) of the table (row j*K + k of the profile table) against job (j + 1) mod J of
    the same scenario at its current configuration sel[s, j+1]: the co-location a bin-packing step
    would have produced (BinPack itself is not specified by the paper)."""
    j = np.arange(J)
    partner = (j + 1) % J
    pairs = np.empty((S, J, K, 2), np.int32)
    pairs[..., 0] = (j[:, None] * K + np.arange(K)[None, :])[None, :, :]
    pairs[..., 1] = (partner * K)[None, :, None] + sel[:, partner][:, :, None]
    return pairs.reshape(-1, 2)


@pytest.mark.parametrize("path", ["tensor", "fma"])
def test_outer_loop_matches_oracle(path):
    S, J, K, M, T = 2, 192, 16, 3, 25
    t = W.whatif_batch(scenarios=[2, 9], J=J).table
    rows = W.iac_rows(7, J, K)
    model = W.iac_model(7, 64)
    gamma0, alpha = 0.02, 0.5
    tau_base = np.full(S * J, 1.15)

    s = esp.Solver(t)
    pred = esp.Predictor(model, path=iac_t.PATHS[path])
    lam_gpu = np.zeros((S, t.P))
    lam_ref = [np.zeros(t.P) for _ in range(S)]
    pen_ref = {}
    for m in range(M):
        sol = s.solve(0.02, T, lambda0=lam_gpu)
        ref = [oracle.solve_scenario(tm, sc, 0.02, T, lambda0=lam_ref[sc])
               for sc, tm in enumerate([W.OptionTable(**{**t.__dict__, **pen_ref})] * S)]
        for sc in range(S):
            assert np.array_equal(sol.sel[sc], ref[sc].sel), (m, sc)
            assert np.array_equal(sol.lam[sc], ref[sc].lam), (m, sc)
        lam_gpu = sol.lam.copy()
        lam_ref = [r.lam.copy() for r in ref]
        # IAC: every option against its partner's current configuration
        pairs = colocation_pairs(S, J, K, sol.sel)
        s_hat32 = pred.predict(rows, pairs, W.IAC_C_MEM)
        want = iac_oracle.predict(rows, pairs, W.IAC_C_MEM, iac_t.as_oracle_model(model))
        bound = iac_t.error_bound(rows, pairs, W.IAC_C_MEM, model, path)
        assert np.all(np.abs(s_hat32.astype(np.float64) - want) <= bound)
        s_hat = s_hat32.astype(np.float64)
        # thresholds from the GPU share in use (Eq. adaptive_threshold), then Gamma for the next round
        util = float(sol.demand[:, 0].sum() / t.capacity[:, 0].sum())
        tau = esp.esp_adaptive_threshold(tau_base, 0.3, util, 0.8, 0.2)
        c_cur = sol.sel.reshape(-1).astype(np.int32)
        esp.esp_set_penalties(s.ctx, gamma0=gamma0, c_cur=c_cur, alpha=alpha, s_hat=s_hat, tau=tau)
        pen_ref = {"values": oracle.penalized_values(t, gamma0, c_cur, alpha, s_hat, tau)}
        assert (s_hat > tau[np.repeat(np.arange(S * J), K)]).any()      # some options are penalised
    pred.close()
    s.close()
