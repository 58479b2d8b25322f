// Device arithmetic shared by the streaming evaluation kernels and the cluster-resident kernel of
// the ESP tatonnement (Sec. 3.2 of the paper). Everything that decides a result bit (the price
// step, the effective prices, the fp32 screen and its bound, the order of fp64 scores) lives here
// once, so both paths compute identical bits.
#pragma once

#include <cmath>
#include <cstdint>
#include <cuda_runtime.h>

#include "esp_common.h"

namespace esp {

constexpr unsigned FULL = 0xffffffffu;
constexpr int kIdxNone = 0x7fffffff;

__device__ __forceinline__ uint32_t smem_u32(const void *p)
{
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

// SplitMix64 finaliser; the per-round selection fingerprint of a scenario is the wrapping sum of
// splitmix64_mix((j << 32) | c_j) over its jobs j.
__device__ __forceinline__ uint64_t splitmix64_mix(uint64_t z)
{
    z = (z ^ (z >> 30)) * 0xbf58476d1ce4e5b9ULL;
    z = (z ^ (z >> 27)) * 0x94d049bb133111ebULL;
    return z ^ (z >> 31);
}

// fp32 value of v truncated toward zero (relative error < 2^-23) for 2^-100 <= |v| <= 2^100, and 0
// (absolute error < 2^-100) below; integer ops only (a double-to-float conversion would run on the
// fp64 pipe). Scenarios with larger values are evaluated exactly and never use the result.
__device__ __forceinline__ float f32_of_f64(double v)
{
    const uint32_t hi = (uint32_t)__double2hiint(v);
    const uint32_t lo = (uint32_t)__double2loint(v);
    // rebase the exponent (1023 -> 127); the sign bit is untouched for |v| >= 2^-127
    const uint32_t t = hi - (896u << 20);
    // 8 exponent and 23 mantissa bits; bit 31 comes out 0 because the rebased exponent is < 256
    const uint32_t bits = __funnelshift_l(lo, t, 3) | (hi & 0x80000000u);
    return ((hi << 1) >= (923u << 21)) ? __uint_as_float(bits) : 0.0f;
}

// Exact fp32 value of a unit count: 2^23 + u is exact in fp32 for 0 <= u < 2^23, so one OR and one
// subtraction replace the int-to-float conversion; larger tables use the conversion instruction.
__device__ __forceinline__ float f32_of_units(int32_t u, bool small)
{
    return small ? (__uint_as_float(0x4b000000u | (uint32_t)u) - 8388608.0f) : __int2float_rn(u);
}

// The fp32 value used by the screen: truncated by integer ops, or (ESP_V32_HW) rounded by the
// conversion instruction; both are within 2^-23 relative (or 2^-100 absolute) of v in range.
__device__ __forceinline__ float screen_value(double v)
{
#if ESP_V32_HW
    return __double2float_rn(v);
#else
    return f32_of_f64(v);
#endif
}

// Signed-integer key with the order of the doubles (no NaN occurs); -0.0 and +0.0 share key 0.
__device__ __forceinline__ long long order_key(double x)
{
    long long b = __double_as_longlong(x);
    if ((b << 1) == 0)
        b = 0;
    return b ^ ((b >> 63) & 0x7fffffffffffffffLL);
}

__device__ __forceinline__ double key_value(long long k)
{
    return __longlong_as_double(k ^ ((k >> 63) & 0x7fffffffffffffffLL));
}

__device__ __forceinline__ double warp_sum_fixed(double x)
{
#pragma unroll
    for (int d = 16; d >= 1; d >>= 1)
        x += __shfl_xor_sync(FULL, x, d);
    return x;
}

__device__ __forceinline__ double warp_max(double x)
{
#pragma unroll
    for (int d = 16; d >= 1; d >>= 1)
        x = fmax(x, __shfl_xor_sync(FULL, x, d));
    return x;
}

// Step size of update `round` (0-based): eta0 (fixed) or eta0 / sqrt(t) with t = round + 1.
__device__ __forceinline__ double step_size(double eta0, int step, int round)
{
    return step == 1 ? eta0 / sqrt((double)(round + 1)) : eta0;
}

// Eq. price_update for one resource: lambda' = max(0, lambda + eta d), d = U - C (RAW) or
// (U - C) / C (NORMALIZED: the same step on capacity-fraction units), one fused multiply-add.
// Cd = (double)C, converted once by the caller.
__device__ __forceinline__ double price_step(double lam, long long U, long long C, double Cd, double eta, int mode)
{
    double excess = (double)(U - C);
    if (mode == 1)
        excess = excess / Cd;
    const double moved = __fma_rn(eta, excess, lam);
    return moved > 0.0 ? moved : 0.0;
}

// Per-unit price of a resource: lambda (RAW) or lambda / C (NORMALIZED); Cd = (double)C.
__device__ __forceinline__ double effective_price(double lam, double Cd, int mode)
{
    return mode == 1 ? lam / Cd : lam;
}

// Screen bound E of a scenario (fp32, rounded up) from M = max|v| + sum_r max p_r * max u_r, or
// +inf when the scenario must be evaluated in fp64 only.
__device__ __forceinline__ float screen_bound(double M, int R, bool exact)
{
    if (exact || !(M <= 0x1p100))
        return INFINITY;
    const double eb = (4.0 * R + 16.0) * 0x1p-24 * M * (1.0 + 0x1p-20) + 0x1p-99;
    return __double2float_ru(eb);
}

}  // namespace esp
