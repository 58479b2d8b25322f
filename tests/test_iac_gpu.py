"""Parity of the IAC predictor's CUDA path (esp_iac_predict, include/esp_iac.h) with the fp64 oracle
(oracle/iac_oracle.py) on seeded synthetic rows, pairs and models.

Tolerance (the paper fixes no precision; the kernel computes in fp32). With u = 2^-24, per pair:
the pairwise features are computed with at most 3 roundings each (|error| <= 3u X, X the magnitude
of the feature, for the intensity difference the sum of both ratios); the folded parameters
W' = s W and b' = s (b - mean) + beta are fp32 roundings of their fp64 values (u relative); a dot
product of n terms accumulated by fused multiply-adds has |error| <= n u (|b'| + sum |W'| |x|)
to first order; ReLU is 1-Lipschitz. Propagated layer by layer:
    M1 = |b1'| + |W1'| X,                  E1 = |W1'| (3u X) + 40 u M1
    M2 = |b2'| + |W2'| (|h1| + E1),        E2 = |W2'| E1 + (H + 3) u M2
    M3 = |b3|  + |W3|  (|h2| + E2),        E3 = |W3| E2 + (H + 2) u M3
and the final 1 + ReLU(y) adds u (1 + M3). The tensor-core path (hidden layers as tcgen05 MMAs on
a three-term tf32 split, esp_iac.h) differs in the two hidden dot products: each product is within
2^-19 = 32u relative (the dropped low-times-low term and the roundings of the low parts), the
tensor core accumulates 64 products (zero padding included) in fp32 whose additions may truncate
(2u each), layer 1's bias enters as one more product (a column of ones times b1', inside M1) and
layer 2's is added in the epilogue: 40 u and (H + 3) u become 160 u and 200 u. The
test allows twice the bound per pair, and checks that the typical error stays near fp32 rounding.
"""

PATHS = {"tensor": 0, "fma": 1}
DOT = {"tensor": (160, lambda H: 200), "fma": (40, lambda H: H + 3)}
TYPICAL = {"tensor": 256, "fma": 64}

import numpy as np
import pytest

from oracle import iac_oracle as iac
from paper_2608_07971_gb300 import workloads as W

pytestmark = pytest.mark.gpu

U = 2.0 ** -24


@pytest.fixture(scope="module")
def lib():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    from paper_2608_07971_gb300 import build, esp
    build.build()
    return esp.load_library()


def as_oracle_model(m):
    return iac.IacModel(W1=m.W1, b1=m.b1, bn1=m.bn1, W2=m.W2, b2=m.b2, bn2=m.bn2, W3=m.W3, b3=m.b3, eps=m.eps)


def folded(W, b, bn, eps):
    W, b, bn = (np.asarray(a, np.float64) for a in (W, b, bn))
    s = bn[0] / np.sqrt(bn[3] + eps)
    return s[:, None] * W, s * (b - bn[2]) + bn[1]


def error_bound(rows, pairs, c_mem, m, path="fma"):
    """Per-pair bound of |kernel - fp64 oracle| (module docstring)."""
    x = iac.feature_matrix(rows, pairs, c_mem)
    X = np.abs(x)
    r = np.asarray(rows, np.float64)
    ratio = np.where(r[:, 0] == 0.0, 0.0, np.abs(r[:, 2]) / np.where(r[:, 0] == 0.0, 1.0, r[:, 0]))
    X[:, 35] = ratio[pairs[:, 0]] + ratio[pairs[:, 1]]
    H = m.W1.shape[0]
    W1f, b1f = folded(m.W1, m.b1, m.bn1, m.eps)
    W2f, b2f = folded(m.W2, m.b2, m.bn2, m.eps)
    W3 = np.abs(np.asarray(m.W3, np.float64))
    om = as_oracle_model(m)
    h1 = iac.relu(iac.batch_norm(x @ np.asarray(m.W1, np.float64).T + np.asarray(m.b1, np.float64), om.bn1, om.eps))
    h2 = iac.relu(iac.batch_norm(h1 @ np.asarray(m.W2, np.float64).T + np.asarray(m.b2, np.float64), om.bn2, om.eps))
    M1 = np.abs(b1f) + X @ np.abs(W1f).T
    c1, c2 = DOT[path][0], DOT[path][1](H)
    E1 = (3 * U * X) @ np.abs(W1f).T + c1 * U * M1
    M2 = np.abs(b2f) + (np.abs(h1) + E1) @ np.abs(W2f).T
    E2 = E1 @ np.abs(W2f).T + c2 * U * M2
    M3 = abs(float(m.b3)) + (np.abs(h2) + E2) @ W3
    E3 = E2 @ W3 + (H + 2) * U * M3
    return 2.0 * (E3 + U * (1.0 + M3))


def random_model(seed, H):
    rng = np.random.default_rng(seed)
    f32 = lambda a: np.asarray(a, np.float32)
    n_in = 36
    W1 = rng.normal(0, np.sqrt(2.0 / n_in), (H, n_in)) / W.IAC_INPUT_STD
    bn = lambda: f32([rng.uniform(0.5, 2.0, H), rng.normal(0, 0.5, H), rng.normal(0, 1.0, H), rng.uniform(0.1, 3.0, H)])
    return W.IacParams(W1=f32(W1), b1=f32(-(W1 @ W.IAC_INPUT_MEAN) + rng.normal(0, 0.3, H)), bn1=bn(),
                       W2=f32(rng.normal(0, np.sqrt(2.0 / H), (H, H))), b2=f32(rng.normal(0, 0.3, H)), bn2=bn(),
                       W3=f32(np.abs(rng.normal(0, np.sqrt(2.0 / H), H)) * np.where(np.arange(H) % 2 == 0, 1.0, -0.5)),
                       b3=float(np.float32(rng.normal(0.0, 0.1))), eps=1e-5)


def gpu_predict(esp, model, rows, pairs, c_mem, path="tensor"):
    import torch
    dev = torch.device("cuda:0")
    p = esp.Predictor(model, path=PATHS[path])
    try:
        r = torch.from_numpy(np.ascontiguousarray(rows, np.float32)).to(dev)
        q = torch.from_numpy(np.ascontiguousarray(pairs, np.int32)).to(dev)
        out = torch.full((len(pairs),), -7.0, dtype=torch.float32, device=dev)
        p.predict(r, q, c_mem, out)
        esp.esp_iac_synchronize(p.h)
        return out.cpu().numpy().astype(np.float64), esp.esp_iac_last_launch_count(p.h)
    finally:
        p.close()


def check(esp, model, rows, pairs, c_mem, path):
    got, launches = gpu_predict(esp, model, rows, pairs, c_mem, path)
    ref = iac.predict(rows, pairs, c_mem, as_oracle_model(model))
    tol = error_bound(rows, pairs, c_mem, model, path)
    err = np.abs(got - ref)
    bad = np.flatnonzero(~(err <= tol))
    assert bad.size == 0, f"{bad.size} pairs beyond the bound, first {bad[:5]}: got {got[bad[:5]]} ref {ref[bad[:5]]}"
    # the bound is a worst case; a systematic slip far below it (a wrong constant, a dropped small
    # term) still shows in the typical error, which for fp32 stays near a few u
    if len(pairs):
        assert np.median(err / np.maximum(ref, 1.0)) <= TYPICAL[path] * U
    assert launches == (1 if len(pairs) else 0)
    return got, ref


@pytest.mark.parametrize("path", ["tensor", "fma"])
@pytest.mark.parametrize("H", [1, 7, 16, 33, 64])
def test_parity_ragged(lib, H, path):
    from paper_2608_07971_gb300 import esp
    rows = W.iac_rows(11, 64, 8)
    pairs = W.iac_pairs(11, 3, 64, 8)[: 1000 + 37]     # a ragged tail after several tiles
    got, ref = check(esp, random_model(H, H), rows, pairs, W.IAC_C_MEM, path)
    assert (ref > 1.0).any()


def test_parity_several_tiles_per_warpgroup(lib):
    """1,024 tiles of 128 pairs, a ragged last one: on a full grid (152 CTAs x 4 warpgroups) most
    warpgroups of the tensor path run two tiles in turn, the second with the roles of their two
    tensor-memory regions swapped; every pair is checked."""
    from paper_2608_07971_gb300 import esp
    w = W.iac_batch(S=4, J=2048, K=16, H=64, seed=9)
    pairs = w.pairs[: len(w.pairs) - 51]
    got, ref = check(esp, w.model, w.rows, pairs, w.c_mem, "tensor")
    assert (ref > 1.0).mean() > 0.2


@pytest.mark.parametrize("path", ["tensor", "fma"])
def test_parity_synthetic_model(lib, path):
    from paper_2608_07971_gb300 import esp
    w = W.iac_batch(S=2, J=256, K=16, H=64, seed=6)
    got, ref = check(esp, w.model, w.rows, w.pairs, w.c_mem, path)
    assert (ref > 1.0).mean() > 0.2 and (ref == 1.0).mean() > 0.2


@pytest.mark.parametrize("path", ["tensor", "fma"])
def test_hand_example_exact(lib, path):
    from paper_2608_07971_gb300 import esp
    from tests import test_oracle_iac as pins
    g = pins.golden()
    names = ["a", "b", "c"]
    rows = np.asarray([g["jobs"][n]["features"] for n in names], np.float32)
    keys = list(g["predictions_by_hand"])
    pairs = np.asarray([[names.index(pins.PAIR_NAMES[k][0]), names.index(pins.PAIR_NAMES[k][1])] for k in keys],
                       np.int32)
    got, _ = gpu_predict(esp, pins.hand_model(iac, g), rows, pairs, g["c_mem"], path)
    np.testing.assert_array_equal(got, [g["predictions_by_hand"][k]["s_hat"] for k in keys])
    got, _ = gpu_predict(esp, pins.hand_model(iac, g, b3=g["clamped"]["b3"]), rows, pairs, g["c_mem"], path)
    np.testing.assert_array_equal(got, np.ones(len(keys)))


@pytest.mark.parametrize("path", ["tensor", "fma"])
def test_zero_sm_self_pairs_and_equal_rows(lib, path):
    from paper_2608_07971_gb300 import esp
    rows = W.iac_rows(12, 16, 4)
    rows[3, 0] = 0.0            # SM Active 0
    rows[9, 0] = 0.0
    rows[10] = rows[11]         # identical rows
    n = rows.shape[0]
    pairs = np.asarray([(i, j) for i in range(n) for j in (i, 3, 9, 11)], np.int32)
    check(esp, random_model(5, 32), rows, pairs, W.IAC_C_MEM, path)


@pytest.mark.parametrize("path", ["tensor", "fma"])
def test_host_call_matches_device_call(lib, path):
    from paper_2608_07971_gb300 import esp
    rows = W.iac_rows(13, 128, 4)
    pairs = W.iac_pairs(13, 2, 128, 4)
    model = random_model(9, 48)
    dev, _ = gpu_predict(esp, model, rows, pairs, W.IAC_C_MEM, path)
    p = esp.Predictor(model, path=PATHS[path])
    try:
        host = p.predict(rows, pairs, W.IAC_C_MEM).astype(np.float64)
        assert esp.esp_iac_last_launch_count(p.h) == 1
        np.testing.assert_array_equal(host, dev)
        assert p.predict(rows, pairs[:0], W.IAC_C_MEM).shape == (0,)
        assert esp.esp_iac_last_launch_count(p.h) == 0
        with pytest.raises(esp.EspError):
            p.predict(rows, np.asarray([[0, rows.shape[0]]], np.int32), W.IAC_C_MEM)
    finally:
        p.close()


@pytest.mark.parametrize("path", ["tensor", "fma"])
def test_out_of_range_pairs_give_nan_on_device(lib, path):
    from paper_2608_07971_gb300 import esp
    rows = W.iac_rows(14, 8, 2)
    pairs = np.asarray([[0, 1], [-1, 0], [3, 16], [16, 3], [5, 5]], np.int32)
    got, _ = gpu_predict(esp, random_model(2, 16), rows, pairs, W.IAC_C_MEM, path)
    assert np.isnan(got[1:4]).all()
    ok = [0, 4]
    ref = iac.predict(rows, pairs[ok], W.IAC_C_MEM, as_oracle_model(random_model(2, 16)))
    assert np.all(np.abs(got[ok] - ref) <= error_bound(rows, pairs[ok], W.IAC_C_MEM, random_model(2, 16), path))


@pytest.mark.parametrize("path", ["tensor", "fma"])
def test_empty_batch_launches_nothing(lib, path):
    from paper_2608_07971_gb300 import esp
    got, launches = gpu_predict(esp, random_model(3, 8), W.iac_rows(1, 4, 2), np.zeros((0, 2), np.int32), 1.0, path)
    assert got.shape == (0,) and launches == 0


def test_invalid_models_rejected(lib):
    from paper_2608_07971_gb300 import esp
    p = esp.Predictor()
    try:
        with pytest.raises(esp.EspError):        # predict before a model
            p.predict(W.iac_rows(1, 2, 2), np.zeros((1, 2), np.int32), 1.0)
        good = random_model(4, 8)
        for field, bad in (("W1", np.full((65, 36), 0.1, np.float32)),
                           ("b2", np.full(8, np.nan, np.float32)),
                           ("bn1", np.vstack([good.bn1[:3], -np.ones((1, 8), np.float32)]))):
            m = W.IacParams(**{**good.__dict__, field: bad})
            if field == "W1":
                m = W.IacParams(**{**good.__dict__, "W1": bad, "b1": np.zeros(65, np.float32)})
            with pytest.raises(esp.EspError):
                p.load(m)
        p.load(good)
        with pytest.raises(esp.EspError):        # c_mem must be positive
            p.predict(W.iac_rows(1, 2, 2), np.zeros((1, 2), np.int32), 0.0)
    finally:
        p.close()


@pytest.mark.parametrize("path", ["tensor", "fma"])
def test_full_batch_sampled(lib, path):
    """The benchmark batch (S=1024 what-if scenarios x 2048 jobs x 16 configurations = 33.5 M pairs,
    H = 64) in one launch; 20,000 sampled pairs against the oracle."""
    import torch
    from paper_2608_07971_gb300 import esp
    w = W.iac_batch()
    dev = torch.device("cuda:0")
    p = esp.Predictor(w.model, path=PATHS[path])
    try:
        r = torch.from_numpy(w.rows).to(dev)
        q = torch.from_numpy(w.pairs).to(dev)
        out = torch.empty(len(w.pairs), dtype=torch.float32, device=dev)
        p.predict(r, q, w.c_mem, out)
        esp.esp_iac_synchronize(p.h)
        idx = np.random.default_rng(0).choice(len(w.pairs), 20000, replace=False)
        idx = np.concatenate([idx, [0, len(w.pairs) - 1]])
        got = out[torch.from_numpy(idx).to(dev)].cpu().numpy().astype(np.float64)
        ref = iac.predict(w.rows, w.pairs[idx], w.c_mem, as_oracle_model(w.model))
        tol = error_bound(w.rows, w.pairs[idx], w.c_mem, w.model, path)
        assert np.all(np.abs(got - ref) <= tol)
        assert np.median(np.abs(got - ref) / ref) <= TYPICAL[path] * U
        assert torch.isfinite(out).all() and bool((out >= 1.0).all())
    finally:
        p.close()
