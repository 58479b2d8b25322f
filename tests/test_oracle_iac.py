"""Pins of the IAC oracle (Sec. 3.3.1 features, Sec. 3.3.2 network and Eq. dnn_pred) against what
does not come from the oracle itself: the hand-worked dyadic example in tests/golden/iac_hand.json,
PyTorch's own Linear / BatchNorm1d (eval) / ReLU / Dropout (eval) layers in fp64, and the invariants
S_hat >= 1 and the symmetry of the pairwise block. Every check takes the oracle module as an
argument, so test_oracle_iac_mutants can run the same checks on planted mistakes."""

import json
import os

import numpy as np
import pytest

from oracle import iac_oracle

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "iac_hand.json")
PAIR_NAMES = {"a|b": ("a", "b"), "b|a": ("b", "a"), "a|a": ("a", "a"), "b|b": ("b", "b"),
              "a|c": ("a", "c"), "b|c": ("b", "c"), "c|c": ("c", "c")}


def golden():
    with open(GOLDEN) as f:
        return json.load(f)


def hand_model(iac, g, b3=None):
    m = g["model"]
    H = m["H"]
    W1 = np.zeros((H, iac.N_FEAT), np.float32)
    for row, col, val in m["W1_nonzero"]:
        W1[row, col] = val
    bn = lambda d: np.asarray([d["gamma"], d["beta"], d["mean"], d["var"]], np.float32)
    return iac.IacModel(W1=W1, b1=np.asarray(m["b1"], np.float32), bn1=bn(m["bn1"]),
                        W2=np.asarray(m["W2"], np.float32), b2=np.asarray(m["b2"], np.float32), bn2=bn(m["bn2"]),
                        W3=np.asarray(m["W3"], np.float32), b3=float(m["b3"] if b3 is None else b3),
                        eps=float(m["eps"]))


# typical magnitude of each feature of random_jobs' pairs, so that W1 x stays of order one
FEATURE_SCALE = np.asarray([1, 1, 1, 40000, 1, 1, 22, 5, 2, 2, 2, 1, 1, 1] * 2 + [1, 1, 1, 1, 1, 1, 1, 5], np.float64)


def random_model(iac, rng, H, eps=1e-5):
    f32 = lambda a: np.asarray(a, np.float32)
    bn = lambda: f32([rng.uniform(0.5, 2.0, H), rng.normal(0, 0.5, H), rng.normal(0, 1.0, H), rng.uniform(0.1, 3.0, H)])
    W1 = rng.normal(0, 0.3, (H, iac.N_FEAT)) / FEATURE_SCALE
    return iac.IacModel(W1=f32(W1), b1=f32(rng.normal(0, 0.5, H)), bn1=bn(),
                        W2=f32(rng.normal(0, 0.3, (H, H))), b2=f32(rng.normal(0, 0.5, H)), bn2=bn(),
                        W3=f32(np.abs(rng.normal(0, 0.3, H)) * np.where(np.arange(H) % 2 == 0, 1.0, -1.0)),
                        b3=float(np.float32(rng.normal(0.0, 0.3))), eps=eps)


def random_jobs(rng, n):
    f = np.zeros((n, 14), np.float32)
    f[:, 0:3] = rng.uniform(0.05, 1.0, (n, 3))
    f[:, 3] = rng.uniform(1000, 80000, n)
    f[:, 4] = rng.uniform(0.0, 1.0, n)
    f[:, 5] = rng.integers(0, 2, n)
    f[:, 6] = rng.uniform(18, 26, n)
    f[:, 7] = rng.uniform(0.1, 10, n)
    f[:, 8:11] = rng.uniform(0, 4, (n, 3))
    f[:, 11:14] = rng.uniform(0, 2, (n, 3))
    return f


# ---- checks (each raises AssertionError on a mismatch)

def check_hand_features(iac):
    g = golden()
    for key, (i, j) in PAIR_NAMES.items():
        fi = np.asarray(g["jobs"][i]["features"], np.float64)
        fj = np.asarray(g["jobs"][j]["features"], np.float64)
        x = iac.pair_features(fi, fj, g["c_mem"])
        assert x.shape == (36,)
        np.testing.assert_array_equal(x[:14], fi, err_msg=key)
        np.testing.assert_array_equal(x[14:28], fj, err_msg=key)
        np.testing.assert_array_equal(x[28:], np.asarray(g["pairwise_by_hand"][key]["values"]), err_msg=key)


def check_hand_predictions(iac):
    g = golden()
    names = ["a", "b", "c"]
    jf = np.asarray([g["jobs"][n]["features"] for n in names], np.float32)
    keys = list(g["predictions_by_hand"])
    pairs = np.asarray([[names.index(PAIR_NAMES[k][0]), names.index(PAIR_NAMES[k][1])] for k in keys], np.int32)
    s = iac.predict(jf, pairs, g["c_mem"], hand_model(iac, g))
    np.testing.assert_array_equal(s, [g["predictions_by_hand"][k]["s_hat"] for k in keys])
    s = iac.predict(jf, pairs, g["c_mem"], hand_model(iac, g, b3=g["clamped"]["b3"]))
    np.testing.assert_array_equal(s, np.ones(len(keys)))


def torch_forward(x, m):
    torch = pytest.importorskip("torch")
    H = m.W1.shape[0]
    t = lambda a: torch.tensor(np.asarray(a, np.float64))
    net = torch.nn.Sequential(
        torch.nn.Linear(36, H), torch.nn.BatchNorm1d(H, eps=m.eps), torch.nn.ReLU(), torch.nn.Dropout(0.2),
        torch.nn.Linear(H, H), torch.nn.BatchNorm1d(H, eps=m.eps), torch.nn.ReLU(), torch.nn.Dropout(0.2),
        torch.nn.Linear(H, 1)).double()
    with torch.no_grad():
        for lin, W, b in ((net[0], m.W1, m.b1), (net[4], m.W2, m.b2), (net[8], np.asarray(m.W3)[None, :], [m.b3])):
            lin.weight.copy_(t(W))
            lin.bias.copy_(t(b))
        for bn, p in ((net[1], m.bn1), (net[5], m.bn2)):
            bn.weight.copy_(t(p[0]))
            bn.bias.copy_(t(p[1]))
            bn.running_mean.copy_(t(p[2]))
            bn.running_var.copy_(t(p[3]))
        net.eval()
        y = net(t(x))[:, 0]
        return (1.0 + torch.relu(y)).numpy()


def check_matches_torch_layers(iac, seed=0, H=16, n=300):
    rng = np.random.default_rng(seed)
    m = random_model(iac, rng, H)
    jf = random_jobs(rng, 40)
    pairs = rng.integers(0, 40, (n, 2)).astype(np.int32)
    x = iac.feature_matrix(jf, pairs, 81920.0)
    s = iac.forward(x, m)
    ref = torch_forward(x, m)
    np.testing.assert_allclose(s, ref, rtol=1e-12, atol=1e-12)
    assert (ref > 1.0).any() and (ref == 1.0).any(), "the case should exercise both sides of the output ReLU"


def check_invariants(iac, seed=1, n=200):
    rng = np.random.default_rng(seed)
    m = random_model(iac, rng, 8)
    jf = random_jobs(rng, 30)
    jf[3, 0] = 0.0                       # one job with SM Active 0
    pairs = rng.integers(0, 30, (n, 2)).astype(np.int32)
    pairs[0] = (3, 7)
    x = iac.feature_matrix(jf, pairs, 81920.0)
    xs = iac.feature_matrix(jf, pairs[:, ::-1], 81920.0)
    np.testing.assert_array_equal(x[:, 28:], xs[:, 28:])        # pairwise block symmetric in (i, j)
    np.testing.assert_array_equal(x[:, :14], xs[:, 14:28])      # per-job blocks swap
    assert np.all(np.isfinite(x))
    assert np.all((x[:, 34] >= 0.0) & (x[:, 34] <= 1.0))
    s = iac.forward(x, m)
    assert np.all(s >= 1.0)


CHECKS = [check_hand_features, check_hand_predictions, check_matches_torch_layers, check_invariants]


def test_hand_features():
    check_hand_features(iac_oracle)


def test_hand_predictions():
    check_hand_predictions(iac_oracle)


@pytest.mark.parametrize("seed,H", [(0, 16), (0, 64), (5, 64)])
def test_matches_torch_layers(seed, H):
    check_matches_torch_layers(iac_oracle, seed, H)


def test_invariants():
    check_invariants(iac_oracle)
