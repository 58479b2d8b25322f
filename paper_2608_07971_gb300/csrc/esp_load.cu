// Load-time kernels of the ESP solver: validation of a table with its per-scenario maxima, the
// marking of exact duplicate options, the sorted layout's gather, and the effective values of the
// Gamma term (esp_set_penalties).

#include <algorithm>
#include <cmath>
#include <cstdint>
#include <cuda_runtime.h>

#include "esp_device.cuh"
#include "esp_kernels.h"

namespace esp {

namespace {

// ---------------------------------------------------------------------------------------------
// Load-time marking of exact duplicates: option o of a job is marked (sign bit of its column-0
// unit) when an earlier option of the same job has the same units, value and group. Such an option
// ties its twin in every round and loses the tie on index, so it never changes a best response;
// the screen skips it. One warp per job, jobs of up to kDedupMaxK options (larger jobs stay
// unmarked and are still exact: the resolution also compares survivors with the first one).

constexpr int kDedupMaxK = 1024;
constexpr int kDedupWarps = 4;

__device__ __forceinline__ uint64_t option_hash(const DevTable &t, int64_t o)
{
    uint64_t h = splitmix64_mix((uint64_t)__double_as_longlong(t.values[o]));
    for (int r = 0; r < t.R; ++r)
        h = splitmix64_mix(h ^ (uint64_t)(uint32_t)(t.units[o * t.R + r] & 0x7fffffff) ^ ((uint64_t)r << 40));
    if (t.group)
        h = splitmix64_mix(h ^ ((uint64_t)t.group[o] << 48));
    return h;
}

__device__ __forceinline__ bool same_option(const DevTable &t, int64_t a, int64_t b)
{
    if (__double_as_longlong(t.values[a]) != __double_as_longlong(t.values[b]))
        return false;
    if (t.group && t.group[a] != t.group[b])
        return false;
    for (int r = 0; r < t.R; ++r)
        if ((t.units[a * t.R + r] & 0x7fffffff) != (t.units[b * t.R + r] & 0x7fffffff))
            return false;
    return true;
}

// kmax: the largest option count marked (<= kDedupMaxK); each warp's hash row is kmax long, so a
// table of small jobs keeps many blocks per SM.
__global__ void __launch_bounds__(kDedupWarps * 32) k_mark_duplicates(DevTable t, int32_t *units,
                                                                     unsigned long long *marked, int kmax)
{
    extern __shared__ uint64_t hs_all[];
    const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
    uint64_t *hs_w = hs_all + (size_t)wid * kmax;
    const int64_t n_jobs = (int64_t)t.S * t.J;
    unsigned int n_marked = 0;   // counted per lane, one atomic per warp at the end
    for (int64_t j = (int64_t)blockIdx.x * kDedupWarps + wid; j < n_jobs; j += (int64_t)gridDim.x * kDedupWarps) {
        const int64_t a = t.job_off[j];
        const int K = (int)(t.job_off[j + 1] - a);
        if (K < 2 || K > kmax)
            continue;
        for (int k = lane; k < K; k += 32)
            hs_w[k] = option_hash(t, a + k);
        __syncwarp();
        for (int k = lane; k < K; k += 32) {
            const uint64_t h = hs_w[k];
            for (int k2 = 0; k2 < k; ++k2) {
                if (hs_w[k2] == h && same_option(t, a + k, a + k2)) {
                    units[(a + k) * t.R] |= (int32_t)0x80000000;
                    ++n_marked;
                    break;
                }
            }
        }
        __syncwarp();
    }
    n_marked = __reduce_add_sync(FULL, n_marked);
    if (lane == 0 && n_marked != 0)
        atomicAdd(marked, (unsigned long long)n_marked);
}

// Sorted layout: one warp per job copies the job's options from the original table and writes its
// padding (units 0 with the duplicate mark on column 0, value 0), so padding never wins.
__global__ void k_gather_sorted(DevTable orig, DevTable sorted, int32_t *units, double *values)
{
    const int lane = threadIdx.x & 31;
    const int64_t n_jobs = (int64_t)sorted.S * sorted.J;
    const int R = sorted.R;
    for (int64_t j = (int64_t)blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5); j < n_jobs;
         j += (int64_t)gridDim.x * (blockDim.x >> 5)) {
        const int64_t dst = sorted.job_off[j];
        const int kp = (int)(sorted.job_off[j + 1] - dst);
        const int64_t oj = sorted.jmap[j];
        const int64_t src = orig.job_off[oj];
        const int k = (int)(orig.job_off[oj + 1] - src);
        for (int i = lane; i < kp * R; i += 32) {
            const int o = i / R, r = i - o * R;
            int32_t u = 0;
            if (o < k)
                u = orig.units[(src + o) * R + r];
            else if (r == 0)
                u = (int32_t)0x80000000;
            units[dst * R + i] = u;
        }
        for (int o = lane; o < kp; o += 32)
            values[dst + o] = (o < k) ? orig.values[src + o] : 0.0;
    }
}

// Gamma term of Eq. esp_score folded into the values (one warp per job): v' = v0 - Gamma with
// Gamma = (c != c_cur ? gamma0 : 0) + alpha * max(0, s_hat - tau), every step one correctly rounded
// fp64 operation (no contraction), so v' is the oracle's to the bit. Flags a current configuration
// outside its job or a non-finite result.
__global__ void k_apply_penalties(DevTable t, const double *values0, const int32_t *c_cur, const double *s_hat,
                                  const double *tau, double gamma0, double alpha, double *values,
                                  unsigned int *flags)
{
    const int lane = threadIdx.x & 31;
    const int64_t n_jobs = (int64_t)t.S * t.J;
    for (int64_t j = (int64_t)blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5); j < n_jobs;
         j += (int64_t)gridDim.x * (blockDim.x >> 5)) {
        const int64_t a = t.job_off[j];
        const int K = (int)(t.job_off[j + 1] - a);
        const int32_t cur = c_cur ? c_cur[j] : -1;
        if (lane == 0 && cur >= K)
            atomicOr(flags, VAL_PENALTY);
        const double tj = s_hat ? tau[j] : 0.0;
        for (int c = lane; c < K; c += 32) {
            const double sw = (cur >= 0 && c != cur) ? gamma0 : 0.0;
            double excess = s_hat ? __dsub_rn(s_hat[a + c], tj) : 0.0;
            if (excess < 0.0)
                excess = 0.0;
            const double gamma = __dadd_rn(sw, __dmul_rn(alpha, excess));
            const double v = __dsub_rn(values0[a + c], gamma);
            if (!isfinite(v))
                atomicOr(flags, VAL_PENALTY);
            values[a + c] = v;
        }
    }
}

// Clears the load-time duplicate marks (sign bit of each option's column-0 unit).
__global__ void k_clear_marks(int32_t *units, int64_t n_opt, int R)
{
    for (int64_t o = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; o < n_opt; o += (int64_t)gridDim.x * blockDim.x)
        units[o * R] &= 0x7fffffff;
}

// Final objectives: primal = sum of chosen values, dual g(lambda) at the final prices, feasibility.

// ---------------------------------------------------------------------------------------------
// Load-time validation and per-scenario maxima (max |v|, max unit per column).

constexpr int kValidateThreads = 256;

// Per scenario (blockIdx.y): finite values, non-negative units, groups in range, and the maxima
// max |v| and max u_r, reduced per warp and per block before one atomic per block and quantity.
__global__ void __launch_bounds__(kValidateThreads) k_validate_options(DevTable t, double *vmax, int32_t *umax,
                                                                       unsigned int *flags)
{
    __shared__ unsigned long long s_vm[kValidateThreads / 32];
    __shared__ int32_t s_um[kValidateThreads / 32][kMaxR];
    __shared__ unsigned int s_bad[kValidateThreads / 32];
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int R = t.R;
    for (int s = blockIdx.y; s < t.S; s += gridDim.y) {
        const int64_t a = t.job_off[(int64_t)s * t.J];
        const int64_t b = t.job_off[(int64_t)(s + 1) * t.J];
        unsigned long long vm = 0ull;   // non-negative doubles order like their bit patterns
        int32_t um[kMaxR];
        for (int r = 0; r < kMaxR; ++r)
            um[r] = 0;
        unsigned int bad = 0;
        for (int64_t o = a + (int64_t)blockIdx.x * blockDim.x + threadIdx.x; o < b;
             o += (int64_t)gridDim.x * blockDim.x) {
            const double v = t.values[o];
            if (!isfinite(v))
                bad |= VAL_VALUE_NONFINITE;
            else
                vm = max(vm, (unsigned long long)__double_as_longlong(fabs(v)));
            for (int r = 0; r < R; ++r) {
                const int32_t u = t.units[o * R + r];
                if (u < 0)
                    bad |= VAL_UNITS_NEG;
                um[r] = max(um[r], u);
            }
            if (t.group && (int)t.group[o] >= t.n_groups)
                bad |= VAL_GROUP_RANGE;
        }
#pragma unroll
        for (int d = 16; d >= 1; d >>= 1)
            vm = max(vm, __shfl_xor_sync(FULL, vm, d));
        bad = __reduce_or_sync(FULL, bad);
        for (int r = 0; r < R; ++r)
            um[r] = __reduce_max_sync(FULL, um[r]);
        if (lane == 0) {
            s_vm[warp] = vm;
            s_bad[warp] = bad;
            for (int r = 0; r < R; ++r)
                s_um[warp][r] = um[r];
        }
        __syncthreads();
        if (threadIdx.x == 0) {
            for (int w = 1; w < kValidateThreads / 32; ++w) {
                vm = max(vm, s_vm[w]);
                bad |= s_bad[w];
            }
            if (bad)
                atomicOr(flags, bad);
            atomicMax(reinterpret_cast<unsigned long long *>(vmax + s), vm);
        }
        if (threadIdx.x < R) {
            int32_t m = s_um[0][threadIdx.x];
            for (int w = 1; w < kValidateThreads / 32; ++w)
                m = max(m, s_um[w][threadIdx.x]);
            atomicMax(umax + (size_t)s * R + threadIdx.x, m);
        }
        __syncthreads();
    }
}

__global__ void k_validate_offsets(DevTable t, unsigned int *flags)
{
    const int64_t n = (int64_t)t.S * t.J;
    unsigned int bad = 0;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x) {
        const int64_t k = t.job_off[i + 1] - t.job_off[i];
        if (k < 1 || k > 0x7fffffffLL)
            bad |= VAL_OFFSETS;
    }
    if (blockIdx.x == 0 && threadIdx.x == 0) {
        if (t.job_off[0] != 0 || t.job_off[n] != t.n_opt)
            bad |= VAL_OFFSETS;
    }
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < (int64_t)t.S * t.P;
         i += (int64_t)gridDim.x * blockDim.x)
        if (t.cap[i] <= 0)
            bad |= VAL_CAPACITY;
    if (bad)
        atomicOr(flags, bad);
}

}  // namespace

cudaError_t launch_validate(const DevTable &t, double *vmax, int32_t *umax, unsigned int *flags, cudaStream_t stream)
{
    if (t.S > 0) {
        // about 8 options per thread, so each block's reduction and atomics cover a few thousand
        const int64_t per = t.n_opt / (t.S > 0 ? t.S : 1) + 1;
        int gx = (int)((per + 8 * kValidateThreads - 1) / (8 * kValidateThreads));
        gx = gx < 1 ? 1 : (gx > 256 ? 256 : gx);
        dim3 grid(gx, t.S < 65535 ? t.S : 65535);
        k_validate_options<<<grid, kValidateThreads, 0, stream>>>(t, vmax, umax, flags);
    }
    k_validate_offsets<<<256, 256, 0, stream>>>(t, flags);
    return cudaGetLastError();
}

cudaError_t launch_gather_sorted(const DevTable &orig, const DevTable &sorted, int32_t *units, double *values,
                                 cudaStream_t stream)
{
    const int64_t n_jobs = (int64_t)sorted.S * sorted.J;
    if (n_jobs == 0)
        return cudaSuccess;
    const int64_t blocks = std::min<int64_t>((n_jobs + 7) / 8, 1 << 20);
    k_gather_sorted<<<(int)blocks, 256, 0, stream>>>(orig, sorted, units, values);
    return cudaGetLastError();
}

cudaError_t launch_apply_penalties(const DevTable &t, const double *values0, const int32_t *c_cur, const double *s_hat,
                                   const double *tau, double gamma0, double alpha, double *values, unsigned int *flags,
                                   cudaStream_t stream)
{
    const int64_t n_jobs = (int64_t)t.S * t.J;
    if (n_jobs == 0)
        return cudaSuccess;
    const int64_t blocks = std::min<int64_t>((n_jobs + 7) / 8, 1 << 20);
    k_apply_penalties<<<(int)blocks, 256, 0, stream>>>(t, values0, c_cur, s_hat, tau, gamma0, alpha, values, flags);
    return cudaGetLastError();
}

cudaError_t launch_clear_marks(int32_t *units, int64_t n_opt, int R, cudaStream_t stream)
{
    if (n_opt == 0)
        return cudaSuccess;
    const int64_t blocks = std::min<int64_t>((n_opt + 255) / 256, 1 << 20);
    k_clear_marks<<<(int)blocks, 256, 0, stream>>>(units, n_opt, R);
    return cudaGetLastError();
}

cudaError_t launch_mark_duplicates(const DevTable &t, int32_t *units, unsigned long long *marked, cudaStream_t stream,
                                   int64_t max_k)
{
    const int64_t n_jobs = (int64_t)t.S * t.J;
    if (n_jobs == 0 || max_k < 2)
        return cudaSuccess;
    const int kmax = (int)std::min<int64_t>(max_k, kDedupMaxK);
    const size_t smem = (size_t)kDedupWarps * kmax * sizeof(uint64_t);
    cudaError_t e = cudaFuncSetAttribute(k_mark_duplicates, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess)
        return e;
    int64_t blocks = (n_jobs + kDedupWarps - 1) / kDedupWarps;
    if (blocks > 65536)
        blocks = 65536;
    k_mark_duplicates<<<(int)blocks, kDedupWarps * 32, smem, stream>>>(t, units, marked, kmax);
    return cudaGetLastError();
}

// One warp per tile: the tile's units (n R int32, duplicate marks included) then its values (n fp64)
// at byte opt_begin * (4R + 8) of the interleaved copy. f32: each unit is written as the bit pattern
// of its fp32 value (exact below 2^24), the duplicate mark kept as the sign bit.
__global__ void k_interleave(DevTable t, const TileDesc *tiles, int64_t n_tiles, unsigned char *il, int f32)
{
    const int lane = threadIdx.x & 31;
    const int64_t warps = (int64_t)gridDim.x * (blockDim.x >> 5);
    const int R = t.R;
    const int64_t W = 4 * R + 8;
    for (int64_t k = (int64_t)blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5); k < n_tiles; k += warps) {
        const TileDesc d = tiles[k];
        int32_t *u = reinterpret_cast<int32_t *>(il + d.opt_begin * W);
        double *v = reinterpret_cast<double *>(il + d.opt_begin * W + (int64_t)d.n_opt * R * 4);
        const int32_t *su = t.units + d.opt_begin * R;
        const double *sv = t.values + d.opt_begin;
        for (int64_t i = lane; i < (int64_t)d.n_opt * R; i += 32) {
            const int32_t x = su[i];
            u[i] = f32 ? (int32_t)(((uint32_t)x & 0x80000000u) |
                                   (uint32_t)__float_as_int(__int2float_rn(x & 0x7fffffff)))
                       : x;
        }
        for (int i = lane; i < d.n_opt; i += 32)
            v[i] = sv[i];
    }
}

cudaError_t launch_interleave(const DevTable &t, const TileDesc *tiles, int64_t n_tiles, unsigned char *il,
                              bool f32, cudaStream_t stream)
{
    if (n_tiles <= 0)
        return cudaSuccess;
    const int64_t blocks = std::min<int64_t>((n_tiles + 7) / 8, 65536);
    k_interleave<<<(int)blocks, 256, 0, stream>>>(t, tiles, n_tiles, il, f32 ? 1 : 0);
    return cudaGetLastError();
}

}  // namespace esp
