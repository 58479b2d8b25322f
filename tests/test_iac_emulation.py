"""The CUDA-core IAC kernel's arithmetic, restated on the CPU with exact fp32 rounding, stays within
the per-pair error bound that the GPU parity tests use (no GPU).

The restatement follows the kernel step by step: Batch Normalization folded in fp64 and rounded
once to fp32 (W' = s W, b' = s (b - mean) + beta, s = gamma / sqrt(var + eps)); the pairwise
features with fp32 additions, products and divisions; each hidden unit accumulated from its bias by
fused multiply-adds over the inputs in order (an fp32 fma emulated exactly through fp64 with an
error-free sum); ReLU; the output accumulated from b3 by fused multiply-adds over the hidden units in
order; 1 + ReLU(y). Compared with the fp64 oracle, every pair lies within the bound derived in
tests/test_iac_gpu.py (a worst case: the largest error seen is 1e-4 to 4e-3 of it), and the
median relative error stays within a few fp32 units of roundoff, the sharper of the two checks the
GPU tests also make."""

import numpy as np
import pytest

from oracle import iac_oracle as iac
from paper_2608_07971_gb300 import workloads as W
from tests import test_iac_gpu as gpu_t
from tests.test_screen_bound import fma32

F32 = np.float32
U = 2.0 ** -24


def fold32(Wm, b, bn, eps):
    Wm, b, bn = (np.asarray(a, np.float32).astype(np.float64) for a in (Wm, b, bn))
    s = bn[0] / np.sqrt(bn[3] + eps)
    return (s[:, None] * Wm).astype(F32), (s * (b - bn[2]) + bn[1]).astype(F32)


def features32(rows, pairs, c_mem):
    a = rows[pairs[:, 0]].astype(F32)
    b = rows[pairs[:, 1]].astype(F32)
    x = np.zeros((len(pairs), 36), F32)
    x[:, :14], x[:, 14:28] = a, b
    half = F32(0.5)
    for k, m in enumerate((0, 1, 2, 4)):
        x[:, 28 + k] = (a[:, m] + b[:, m]) * half
    x[:, 32] = a[:, 5] + b[:, 5]
    x[:, 33] = (a[:, 3] + b[:, 3]) / F32(c_mem)
    lo, hi = np.minimum(a[:, 0], b[:, 0]), np.maximum(a[:, 0], b[:, 0])
    with np.errstate(divide="ignore", invalid="ignore"):
        x[:, 34] = np.where(hi == 0, F32(1.0), lo / np.where(hi == 0, F32(1.0), hi))
        ia = np.where(a[:, 0] == 0, F32(0.0), a[:, 2] / np.where(a[:, 0] == 0, F32(1.0), a[:, 0]))
        ib = np.where(b[:, 0] == 0, F32(0.0), b[:, 2] / np.where(b[:, 0] == 0, F32(1.0), b[:, 0]))
    x[:, 35] = np.abs(ia - ib)
    return x


def kernel32(rows, pairs, c_mem, m):
    """Output of the CUDA-core kernel's arithmetic, fp32 throughout."""
    W1f, b1f = fold32(m.W1, m.b1, m.bn1, m.eps)
    W2f, b2f = fold32(m.W2, m.b2, m.bn2, m.eps)
    W3 = np.asarray(m.W3, F32)
    H = W1f.shape[0]
    x = features32(rows, pairs, c_mem)
    n = len(pairs)
    acc = np.broadcast_to(b1f, (n, H)).copy()
    for i in range(36):
        acc = fma32(np.broadcast_to(W1f[:, i], (n, H)), np.broadcast_to(x[:, i:i + 1], (n, H)), acc)
    h1 = np.maximum(acc, F32(0.0))
    acc = np.broadcast_to(b2f, (n, H)).copy()
    for i in range(H):
        acc = fma32(np.broadcast_to(W2f[:, i], (n, H)), np.broadcast_to(h1[:, i:i + 1], (n, H)), acc)
    h2 = np.maximum(acc, F32(0.0))
    y = np.full(n, F32(m.b3), F32)
    for o in range(H):
        y = fma32(np.full(n, W3[o], F32), h2[:, o], y)
    return (F32(1.0) + np.maximum(y, F32(0.0))).astype(np.float64)


def check(m, rows, pairs, c_mem):
    got = kernel32(rows, pairs, c_mem, m)
    ref = iac.predict(rows, pairs, c_mem, gpu_t.as_oracle_model(m))
    tol = gpu_t.error_bound(rows, pairs, c_mem, m, "fma")
    err = np.abs(got - ref)
    assert np.all(err <= tol), np.flatnonzero(err > tol)[:5]
    assert np.median(err / np.maximum(ref, 1.0)) <= 64 * U
    # a worst-case bound: the largest error is a small but visible fraction of it
    assert (err / tol).max() >= 1e-4
    return got, ref


@pytest.mark.parametrize("H", [1, 7, 33, 64])
def test_emulated_kernel_within_bound_ragged_models(H):
    rows = W.iac_rows(11, 64, 8)
    pairs = W.iac_pairs(11, 3, 64, 8)[:1037]
    got, ref = check(gpu_t.random_model(H, H), rows, pairs, W.IAC_C_MEM)
    assert (ref > 1.0).any()


def test_emulated_kernel_within_bound_synthetic_model():
    w = W.iac_batch(S=1, J=128, K=16, H=64, seed=6)
    got, ref = check(w.model, w.rows, w.pairs, w.c_mem)
    assert (ref > 1.0).mean() > 0.2 and (ref == 1.0).mean() > 0.2


def test_emulated_kernel_zero_sm_and_self_pairs():
    rows = W.iac_rows(12, 16, 4)
    rows[3, 0] = 0.0
    rows[9, 0] = 0.0
    rows[10] = rows[11]
    n = rows.shape[0]
    pairs = np.asarray([(i, j) for i in range(n) for j in (i, 3, 9, 11)], np.int32)
    check(gpu_t.random_model(5, 32), rows, pairs, W.IAC_C_MEM)


def test_emulated_kernel_is_exact_on_the_hand_example():
    """The dyadic hand example of the oracle pins is exact in fp32 too."""
    from tests import test_oracle_iac as pins
    g = pins.golden()
    names = ["a", "b", "c"]
    rows = np.asarray([g["jobs"][k]["features"] for k in names], np.float32)
    keys = list(g["predictions_by_hand"])
    pairs = np.asarray([[names.index(pins.PAIR_NAMES[k][0]), names.index(pins.PAIR_NAMES[k][1])] for k in keys],
                       np.int32)
    got = kernel32(rows, pairs, g["c_mem"], pins.hand_model(iac, g))
    np.testing.assert_array_equal(got, [g["predictions_by_hand"][k]["s_hat"] for k in keys])
