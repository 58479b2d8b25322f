"""The tensor-core IAC kernel's arithmetic, restated on the CPU, stays within the per-pair error bound
that the GPU parity tests use for that path (no GPU).

The restatement follows the kernel (include/esp_iac.h, tensor path): the pairwise features in fp32 as
the CUDA-core kernel computes them; layer 1 as D1 = [X | 1 | 0] [W1' | b1' | 0]^T over 40 columns,
the bias entering as the product of a column of ones with b1'; layer 2 as D2 = H1 W2'^T over 64
columns with H1 = ReLU(D1); every operand split into a_hi = a truncated to tf32 and a_lo = the
remainder rounded to the nearest tf32 value (ties away from zero), and each k-step adding
a_hi b_hi, a_hi b_lo and a_lo b_hi, in that order, to an fp32 accumulator; then the epilogue
S_hat = 1 + ReLU(b3 + sum_o w3_o ReLU(D2_o + b2'_o)) in fp32 with fused multiply-adds in order.

Products of two tf32 values are exact in fp32 (11-bit significands). How the tensor core adds them
is not documented, so the accumulator is modelled pessimistically: one addition per product, in issue
order, each truncated toward zero (the error model the bound assumes: 2u per addition). Compared with
the fp64 oracle every pair lies within the bound of tests/test_iac_gpu.py for the tensor path, and the
median error stays within its typical-error check.

That bound is a worst case over the magnitudes of the dot products' terms, and the network's sums
cancel, so on these models it is loose by two to three orders of magnitude; about half of the
outputs are also clamped to exactly 1 by the final ReLU. The typical error is therefore taken here
over the unclamped outputs, where it separates the three-term split (a median of 12-40 units of
fp32 roundoff under the truncating model) from a split that drops the a_lo b_hi products (thousands
of units): the last test plants that mistake and requires the check to fail."""

import numpy as np
import pytest

from oracle import iac_oracle as iac
from paper_2608_07971_gb300 import workloads as W
from tests import test_iac_gpu as gpu_t
from tests.test_iac_emulation import features32, fold32
from tests.test_screen_bound import fma32

F32 = np.float32
U = 2.0 ** -24
K1, K2 = 40, 64


def tf32_hi(a):
    """a truncated to tf32 (the low 13 bits of the fp32 pattern cleared)."""
    return (np.asarray(a, F32).view(np.uint32) & np.uint32(0xFFFFE000)).view(F32)


def tf32_round(a):
    """a rounded to the nearest tf32 value, ties away from zero (magnitude rounding of the pattern)."""
    b = np.asarray(a, F32).view(np.uint32)
    return ((b + np.uint32(0x1000)) & np.uint32(0xFFFFE000)).view(F32)


def split(a):
    hi = tf32_hi(a)
    return hi, tf32_round(np.asarray(a, F32) - hi)   # the fp32 difference is exact


def add_rz(acc, p):
    """fp32 acc + p truncated toward zero, exactly (error-free sum in fp64, then a directed rounding)."""
    a, b = acc.astype(np.float64), p.astype(np.float64)
    s = a + b
    bb = s - a
    e = (a - (s - bb)) + (b - bb)                    # a + b = s + e exactly
    r = s.astype(F32)
    d = r.astype(np.float64) - s                     # exact: r is the fp32 neighbour of s
    over = np.where(s + e > 0, d > e, np.where(s + e < 0, d < e, False))   # |r| > |a + b|
    out = r.copy()
    out[over] = np.nextafter(r[over], F32(0.0))
    return out


SPLIT3 = ((0, 0), (0, 1), (1, 0))   # a_hi b_hi, a_hi b_lo, a_lo b_hi (0: high part, 1: low part)


def contract(A, B, terms=SPLIT3):
    """Split-tf32 product A (n x K) B^T (m x K) with the modelled accumulator, in the kernel's order;
    K is zero-padded to whole k-steps of 8 as in the kernel (a zero product leaves the sum exact)."""
    K = -(-A.shape[1] // 8) * 8
    A = np.pad(np.asarray(A, F32), ((0, 0), (0, K - A.shape[1])))
    B = np.pad(np.asarray(B, F32), ((0, 0), (0, K - B.shape[1])))
    As, Bs = split(A), split(B)
    n, m = A.shape[0], B.shape[0]
    acc = np.zeros((n, m), F32)
    for k0 in range(0, K, 8):                        # one MMA k-step: three MMAs of 8 columns each
        for ia, ib in terms:
            a_part, b_part = As[ia], Bs[ib]
            for k in range(k0, k0 + 8):
                prod = a_part[:, k:k + 1] * b_part[:, k][None, :]     # exact in fp32
                acc = add_rz(acc, prod.astype(F32))
    return acc


def kernel_tc32(rows, pairs, c_mem, m, terms=SPLIT3):
    W1f, b1f = fold32(m.W1, m.b1, m.bn1, m.eps)
    W2f, b2f = fold32(m.W2, m.b2, m.bn2, m.eps)
    W3 = np.asarray(m.W3, F32)
    H = W1f.shape[0]
    x = features32(rows, pairs, c_mem)
    n = len(pairs)
    X = np.zeros((n, K1), F32)
    X[:, :36] = x
    X[:, 36] = F32(1.0)                              # the column that carries layer 1's bias
    B1 = np.zeros((H, K1), F32)
    B1[:, :36] = W1f
    B1[:, 36] = b1f
    h1 = np.maximum(contract(X, B1, terms), F32(0.0))
    d2 = contract(h1, W2f, terms)
    y = np.full(n, F32(m.b3), F32)
    one = np.ones(n, F32)
    for o in range(H):
        t = np.maximum(fma32(one, d2[:, o], np.full(n, b2f[o], F32)), F32(0.0))   # fp32 add, then ReLU
        y = fma32(np.full(n, W3[o], F32), t, y)
    return fma32(one, np.maximum(y, F32(0.0)), one).astype(np.float64)


def check(m, rows, pairs, c_mem, terms=SPLIT3):
    got = kernel_tc32(rows, pairs, c_mem, m, terms)
    ref = iac.predict(rows, pairs, c_mem, gpu_t.as_oracle_model(m))
    tol = gpu_t.error_bound(rows, pairs, c_mem, m, "tensor")
    err = np.abs(got - ref)
    assert np.all(err <= tol), np.flatnonzero(err > tol)[:5]
    assert np.median(err / np.maximum(ref, 1.0)) <= gpu_t.TYPICAL["tensor"] * U
    free = ref > 1.0                                 # outputs the final ReLU does not clamp to 1
    assert np.median(err[free] / ref[free]) <= gpu_t.TYPICAL["tensor"] * U
    assert err.max() > 0.0                           # the restatement is not the fp64 computation
    return got, ref


@pytest.mark.parametrize("H", [1, 7, 33, 64])
def test_emulated_tensor_path_within_bound_ragged_models(H):
    rows = W.iac_rows(11, 64, 8)
    pairs = W.iac_pairs(11, 3, 64, 8)[:600]
    got, ref = check(gpu_t.random_model(H, H), rows, pairs, W.IAC_C_MEM)
    assert (ref > 1.0).any()


def test_emulated_tensor_path_within_bound_synthetic_model():
    w = W.iac_batch(S=1, J=64, K=16, H=64, seed=6)
    got, ref = check(w.model, w.rows, w.pairs, w.c_mem)
    assert (ref > 1.0).mean() > 0.2 and (ref == 1.0).mean() > 0.2


def test_split_is_exact_and_truncating_sum_is_directed():
    """The split reproduces every fp32 value to within its dropped low part, and the modelled addition
    rounds toward zero: against exact sums it never moves away from zero and errs by less than an ulp."""
    rng = np.random.default_rng(3)
    a = (rng.standard_normal(20000) * np.exp2(rng.integers(-20, 20, 20000))).astype(F32)
    hi, lo = split(a)
    assert np.all(tf32_hi(hi) == hi) and np.all(tf32_hi(lo) == lo)
    r = a.astype(np.float64) - hi.astype(np.float64) - lo.astype(np.float64)
    assert np.all(np.abs(r) <= np.abs(a.astype(np.float64)) * 2.0 ** -21)
    b = (rng.standard_normal(20000) * np.exp2(rng.integers(-40, 40, 20000))).astype(F32)
    s = add_rz(a, b).astype(np.float64)
    exact = a.astype(np.float64) + b.astype(np.float64)   # differs from a + b only past 2^-53 relative
    assert np.all(np.abs(s) <= np.abs(exact) * (1 + 2.0 ** -50))
    ulp = np.spacing(np.abs(s).astype(F32)).astype(np.float64)
    assert np.all(np.abs(exact - s) <= ulp * (1 + 2.0 ** -20))
    # a tie on the fp32 grid is truncated, not rounded to even
    t = add_rz(np.array([1.0], F32), np.array([2.0 ** -24 * 3], F32))
    assert t[0] == F32(1.0) + F32(2.0 ** -23)


@pytest.mark.parametrize("H", [7, 64])
def test_dropped_low_times_high_products_fail_the_check(H):
    """A planted mistake: the split without the a_lo b_hi products stays inside the worst-case bound
    but not inside the typical error of the unclamped outputs."""
    rows = W.iac_rows(11, 64, 8)
    pairs = W.iac_pairs(11, 3, 64, 8)[:600]
    with pytest.raises(AssertionError):
        check(gpu_t.random_model(H, H), rows, pairs, W.IAC_C_MEM, terms=((0, 0), (0, 1)))
