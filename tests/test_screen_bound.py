"""The fp32 screen's error bound, checked on the CPU (no GPU).

The evaluation kernels score every option first in fp32,
    q = fma32(p32_{R-1}, u32_{R-1}, ... fma32(p32_0, u32_0, -v32)),
with p32 the prices rounded to fp32, u32 the units converted to fp32 and v32 the value truncated to
fp32 by integer operations (0 below 2^-100), and rely on |q - s| <= E for the fp64 reduced cost s
of Eq. esp_score, with E = (4R + 16) 2^-24 M_s + 2^-99 computed per scenario from
M_s = max|v| + sum_r max p_r max u_r and rounded up to fp32. Each step is restated here with exact
IEEE single-precision rounding (an fp32 fused multiply-add is emulated through fp64 with an
error-free sum, so ties are decided exactly), and E the way the scenario's warp computes it (lane
terms, xor-butterfly sum in fp64). The distance to the exact rational value of s must stay within E
less the fp64 chain's own rounding (R 2^-52 M), on typical, extreme and adversarial inputs."""

import zlib
from fractions import Fraction

import numpy as np
import pytest

TWO = Fraction(2)


def fma32(a, b, c):
    """Correctly rounded fp32 a * b + c for fp32 arrays a, b, c (a * b is exact in fp64)."""
    a, b, c = (np.asarray(x, np.float32).astype(np.float64) for x in (a, b, c))
    t = a * b
    s = t + c
    bb = s - t
    e = (t - (s - bb)) + (c - bb)              # t + c = s + e exactly
    r = s.astype(np.float32)
    rd = r.astype(np.float64)
    up = np.nextafter(r, np.float32(np.inf)).astype(np.float64)
    dn = np.nextafter(r, np.float32(-np.inf)).astype(np.float64)
    # the only ambiguous case: s exactly halfway between two fp32 neighbours, e breaking the tie
    mid_hi = (rd + up) / 2.0
    mid_lo = (rd + dn) / 2.0
    fix_up = (s == mid_hi) & (e > 0)
    fix_dn = (s == mid_lo) & (e < 0)
    out = r.copy()
    out[fix_up] = up[fix_up].astype(np.float32)
    out[fix_dn] = dn[fix_dn].astype(np.float32)
    return out


def v32_of(v):
    """fp32 of v truncated toward zero (24-bit significand); 0 when |v| < 2^-100."""
    bits = np.asarray(v, np.float64).view(np.uint64) & ~np.uint64((1 << 29) - 1)
    t = bits.view(np.float64)
    return np.where(np.abs(v) < 2.0 ** -100, 0.0, t).astype(np.float32)


def screen(units, values, p64):
    """q of every option (rows of units) at fp64 prices p64."""
    p32 = p64.astype(np.float32)
    q = -v32_of(values)
    for r in range(units.shape[1]):
        q = fma32(np.full(len(q), p32[r], np.float32), units[:, r].astype(np.float32), q)
    return q


def bound(units, values, p64):
    """E of the scenario as its warp computes it: lane r's term p_r * max u_r, an xor-butterfly sum
    over 32 lanes in fp64, M = max|v| + sum, then (4R + 16) 2^-24 M (1 + 2^-20) + 2^-99 rounded up
    to fp32."""
    R = units.shape[1]
    x = np.zeros(32)
    x[:R] = p64 * units.max(axis=0).astype(np.float64)
    for d in (16, 8, 4, 2, 1):
        x = x + x[np.arange(32) ^ d]
    M = np.abs(values).max() + x[0]
    eb = (4.0 * R + 16.0) * 2.0 ** -24 * M * (1.0 + 2.0 ** -20) + 2.0 ** -99
    e32 = np.float32(eb)
    if float(e32) < eb:
        e32 = np.nextafter(e32, np.float32(np.inf))
    return float(e32), M


def exact_s(u_row, v, p64):
    s = -Fraction(float(v))
    for r in range(len(u_row)):
        s += Fraction(float(p64[r])) * int(u_row[r])
    return s


def check(units, values, p64, sample=None):
    """Largest |q - s| / (E - R 2^-52 M) over the options (at most `sample` of them, exactly)."""
    q = screen(units, values, p64)
    E, M = bound(units, values, p64)
    R = units.shape[1]
    budget = Fraction(E) - R * Fraction(M) * TWO ** -52
    assert budget > 0
    idx = np.arange(len(values)) if sample is None else np.random.default_rng(0).choice(len(values), sample, False)
    worst = Fraction(0)
    for i in idx:
        d = abs(Fraction(float(q[i])) - exact_s(units[i], values[i], p64))
        worst = max(worst, d / budget)
    return float(worst)


def test_fp32_fma_emulation_is_correctly_rounded():
    """Against exact rationals on random operands and on exact halfway cases: (1 + 2^-23) * 1.5 has
    25 significant bits, so it lies midway between two fp32 numbers; adding 0 leaves the tie to the
    even neighbour, adding +-2^-60 (lost in the fp64 sum, kept in its error term) must round up or
    down."""
    rng = np.random.default_rng(1)
    n = 4000
    a = rng.standard_normal(n).astype(np.float32)
    b = rng.integers(0, 1 << 24, n).astype(np.float32)
    c = (rng.standard_normal(n) * 1e6).astype(np.float32)
    c[:500] = -(a[:500].astype(np.float64) * b[:500].astype(np.float64)).astype(np.float32)   # cancellation
    ties = np.float32(1.0 + 2.0 ** -23), np.float32(1.5)
    a[500:530], b[500:530] = ties
    c[500:510] = 0.0
    c[510:520] = np.float32(2.0 ** -60)
    c[520:530] = np.float32(-2.0 ** -60)
    a[530:540], b[530:540] = -ties[0], ties[1]
    c[530:540] = np.float32(2.0 ** -60)
    got = fma32(a, b, c)
    for i in range(n):
        x = Fraction(float(a[i])) * Fraction(float(b[i])) + Fraction(float(c[i]))
        f = float(x)
        if Fraction(f) == x:
            want = np.float32(f)                # exact in fp64: one rounding to fp32
        else:                                   # the fp32 neighbours, nearest first
            lo = np.float32(f)
            cand = [np.nextafter(lo, np.float32(-np.inf)), lo, np.nextafter(lo, np.float32(np.inf))]
            want = min(cand, key=lambda y: abs(Fraction(float(y)) - x))
        assert got[i] == want, (i, a[i], b[i], c[i])
    t = float(ties[0]) * 1.5                                           # exact in fp64
    assert float(got[500]) == float(np.float32(t))                      # the tie, to even
    assert float(got[510]) > t > float(got[520])                        # decided by the error term
    assert float(got[510]) - float(got[520]) == 2.0 ** -23               # neighbours


def test_value_truncation_and_range():
    v = np.array([1.0, -1.0 - 2.0 ** -30, 3.141592653589793, 2.0 ** -100, 2.0 ** -101, -2.0 ** 100, 0.0])
    got = v32_of(v)
    assert got[0] == 1.0 and got[1] == -1.0 and got[3] == np.float32(2.0 ** -100) and got[4] == 0.0
    assert abs(float(got[2]) - v[2]) < 2.0 ** -22 * v[2] and float(got[2]) <= v[2]
    assert got[5] == np.float32(-2.0 ** 100) and got[6] == 0.0


@pytest.mark.parametrize("case", ["whatif_like", "large_units", "values_near_2e100", "values_near_2em100",
                                  "cancellation", "r16_mixed_scales", "r1", "subnormal_prices"])
def test_screen_within_bound(case):
    rng = np.random.default_rng(zlib.crc32(case.encode()))
    n = 3000
    if case == "whatif_like":
        R = 6
        units = rng.integers(0, 163841, (n, R)).astype(np.int64)
        values = np.exp(rng.standard_normal(n))
        p64 = rng.random(R) * 1e-5
    elif case == "large_units":
        R = 8
        units = rng.integers((1 << 31) - (1 << 20), (1 << 31) - 1, (n, R)).astype(np.int64)
        values = rng.random(n) * 1e9
        p64 = rng.random(R) * 1e-3
    elif case == "values_near_2e100":
        R = 4
        units = rng.integers(0, 1000, (n, R)).astype(np.int64)
        values = (0.5 + 0.5 * rng.random(n)) * 2.0 ** 100
        p64 = rng.random(R) * 2.0 ** 80
    elif case == "values_near_2em100":
        R = 4
        units = rng.integers(0, 1000, (n, R)).astype(np.int64)
        values = rng.random(n) * 2.0 ** -98
        p64 = rng.random(R) * 2.0 ** -110
    elif case == "cancellation":
        # value equal to the rent up to a few ulps: q and s are tiny differences of large terms
        R = 6
        units = rng.integers(1, 1 << 22, (n, R)).astype(np.int64)
        p64 = rng.random(R)
        values = units.astype(np.float64) @ p64 * (1.0 + rng.standard_normal(n) * 1e-15)
    elif case == "r16_mixed_scales":
        R = 16
        units = rng.integers(0, 1 << 24, (n, R)).astype(np.int64)
        values = np.exp(rng.standard_normal(n) * 10)
        p64 = np.exp(rng.standard_normal(R) * 8)
    elif case == "r1":
        R = 1
        units = rng.integers(0, 1 << 31, (n, R)).astype(np.int64)
        values = rng.random(n) * 1e6
        p64 = np.array([rng.random() * 1e-3])
    else:
        R = 5
        units = rng.integers(0, 1 << 20, (n, R)).astype(np.int64)
        values = rng.random(n) * 2.0 ** -90
        p64 = rng.random(R) * 2.0 ** -135      # fp32 subnormals
    worst = check(units, values, p64)
    assert worst <= 1.0, worst
    assert worst <= 0.5 or case in ("cancellation", "values_near_2em100", "subnormal_prices"), worst


def test_bound_is_reached_within_its_stated_margin():
    """Errors aligned on purpose (R = 1): values whose truncation to fp32 drops almost a whole fp32
    ulp (2^-23 |v|), prices just above a midpoint of the fp32 grid (rounded up by 2^-24 p), and a
    rent p u equal to v to within p, so that both errors add with the same sign and the final
    rounding is negligible: |q - s| is close to 3 2^-24 v. With M ~ 2 max v the ratio to
    E = 20 2^-24 M is about 3/40 (0.066 measured), and the derivation's own worst case
    (R + 4) 2^-24 M is 1/4 of E: a bound too small by a factor of 15 would fail here."""
    rng = np.random.default_rng(7)
    n = 3000
    # values at the bottom of the binade [2^20, 2^21), where one fp32 ulp is 2^-23 |v|
    mant = (rng.integers(0, 1 << 10, n).astype(np.uint64) << np.uint64(29)) | np.uint64((1 << 29) - 1)
    values = ((np.uint64(1023 + 20) << np.uint64(52)) | mant).view(np.float64)
    p32 = np.float32(1.0 + rng.integers(0, 1 << 23) * 2.0 ** -23)
    p64 = np.array([float(p32) + 2.0 ** -24 + 2.0 ** -40])                             # rounds up
    assert np.float32(p64[0]) == np.nextafter(p32, np.float32(2))
    units = np.rint(values / p64[0]).astype(np.int64)[:, None]
    worst = check(units, values, p64)
    assert 0.05 <= worst <= 0.25, worst


def test_placement_screen_within_bound():
    """The factored placement screen: the global columns of configuration k scored once,
    g_k = chain over r < rg from -v32_k, then per node n the fp32 sum g_k + pen_n with
    pen_n = fp32(sigma_j * D[a_j][b_n]) (one rounding more than a stored option), then the
    node-priced columns. The fp64 score it must bound is the chain of the expanded option, from
    v_kn = v_k - pen_n rounded to fp64. M takes |v_k| + |sigma_j| max D (1 + 2^-20) as the value
    bound, and for each node-priced column the largest price over the nodes."""
    rng = np.random.default_rng(11)
    J, KC, N, R, rg, NT = 10, 12, 64, 8, 6, 8
    units = rng.integers(0, 200000, (J, KC, R)).astype(np.int64)
    values = np.exp(rng.standard_normal((J, KC)))
    sens = (rng.random(J) * 0.5).astype(np.float32)
    D = rng.beta(2, 8, (NT, NT)).astype(np.float32)
    a = rng.integers(0, NT, J)
    b = rng.integers(0, NT, N)
    P = rg + (R - rg) * N
    p64 = rng.random(P) * 1e-5
    p32 = p64.astype(np.float32)
    dmax = float(D.max())
    vmax = max(float(np.abs(values[j]).max()) + abs(float(sens[j])) * dmax * (1.0 + 2.0 ** -20) for j in range(J))
    umax = units.reshape(-1, R).max(axis=0).astype(np.float64)
    x = np.zeros(32)
    x[:rg] = p64[:rg] * umax[:rg]
    for c2 in range(R - rg):
        x[rg + c2] = p64[rg + c2::R - rg].max() * umax[rg + c2]
    for d in (16, 8, 4, 2, 1):
        x = x + x[np.arange(32) ^ d]
    M = vmax + x[0]
    eb = (4.0 * R + 16.0) * 2.0 ** -24 * M * (1.0 + 2.0 ** -20) + 2.0 ** -99
    E = np.float32(eb)
    if float(E) < eb:
        E = np.nextafter(E, np.float32(np.inf))
    budget = Fraction(float(E)) - R * Fraction(M) * TWO ** -52
    worst = Fraction(0)
    for j in range(J):
        pen = (sens[j] * D[a[j], b]).astype(np.float32)                 # fp32 products, per node
        for k in range(KC):
            g = -v32_of(np.array([values[j, k]]))
            for r in range(rg):
                g = fma32(p32[r:r + 1], units[j, k, r:r + 1].astype(np.float32), g)
            q = (np.full(N, g[0], np.float32) + pen).astype(np.float32)  # fp32 sum, one rounding
            cols = [rg + (R - rg) * np.arange(N) + (r - rg) for r in range(rg, R)]
            for i, r in enumerate(range(rg, R)):
                q = fma32(p32[cols[i]], np.full(N, units[j, k, r], np.float32), q)
            for n in range(N):
                v_kn = float(values[j, k]) - float(pen[n])               # the expanded option's value
                s = -Fraction(v_kn)
                for r in range(R):
                    col = r if r < rg else rg + (R - rg) * n + (r - rg)
                    s += Fraction(float(p64[col])) * int(units[j, k, r])
                worst = max(worst, abs(Fraction(float(q[n])) - s) / budget)
    assert float(worst) <= 0.5, float(worst)


def ru32(x: Fraction) -> np.float32:
    """The smallest fp32 number >= x."""
    c = np.float32(float(x))
    while Fraction(float(c)) < x:
        c = np.nextafter(c, np.float32(np.inf))
    while True:
        d = np.nextafter(c, np.float32(-np.inf))
        if Fraction(float(d)) >= x:
            c = d
        else:
            return c


def resident_bound(p64, umax, vmax, R):
    """E of the cluster-resident kernel: every fp32 operation rounded up (p <= p32 (1 + 2^-23) +
    2^-149, lane terms p_up * max u summed by a 16-lane xor butterfly, M = max|v| + sum, then
    (4R + 16) 2^-24 M + 2^-99); returns 2E / 2."""
    F = lambda v: Fraction(float(v))                                   # noqa: E731
    p32 = p64.astype(np.float32)
    terms = [np.float32(0.0)] * 16
    for r in range(R):
        p_up = ru32(F(ru32(F(p32[r]) * F(np.float32(1.0 + 2.0 ** -23)))) + TWO ** -149)
        terms[r] = ru32(F(p_up) * F(ru32(Fraction(int(umax[r])))))
    for d in (8, 4, 2, 1):
        terms = [ru32(F(terms[i]) + F(terms[i ^ d])) for i in range(16)]
    M = ru32(F(ru32(Fraction(float(vmax)))) + F(terms[0]))
    coef = np.float32((4.0 * R + 16.0) * 2.0 ** -24)
    return F(ru32(F(ru32(F(M) * F(coef))) + TWO ** -99))


@pytest.mark.parametrize("seed", range(6))
def test_bound_computations_never_undercut_the_exact_bound(seed):
    """Both computed bounds (the streaming path's fp64 M with a (1 + 2^-20) factor, rounded up to
    fp32 at the end; the resident path's fp32 arithmetic rounded up at every step) are at least the
    exact (4R + 16) 2^-24 M + 2^-99 with M = max|v| + sum_r p_r max u_r in exact arithmetic."""
    rng = np.random.default_rng(100 + seed)
    checked = 0
    for _ in range(50):
        R = int(rng.integers(1, 17))
        umax = rng.integers(0, 1 << 31, R) if seed % 2 else rng.integers(0, 1 << 18, R)
        p64 = np.exp(rng.standard_normal(R) * (4 + 4 * seed)) * rng.random(R)
        vmax = float(np.exp(rng.standard_normal() * (4 + 4 * seed)))
        M = Fraction(vmax) + sum(Fraction(float(p64[r])) * int(umax[r]) for r in range(R))
        if M > TWO ** 90:
            continue
        exact = (4 * R + 16) * TWO ** -24 * M + TWO ** -99
        units = np.zeros((2, R), np.int64)
        units[0] = umax
        E_stream, _ = bound(units, np.array([vmax, 0.0]), p64)
        assert Fraction(E_stream) >= exact
        assert resident_bound(p64, umax, vmax, R) >= exact
        checked += 1
    assert checked >= 10
