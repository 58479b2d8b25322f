// Allocation-free best response (esp_evaluate_noalloc in include/esp.h).
//
// Some callers cannot allocate device memory at the point where they need a best response: code
// that runs while another framework owns the whole device through its own caching allocator, or a
// scheduler loop that must not block on cudaMalloc / cudaFree (both synchronise the device) and
// works from a fixed memory budget set aside at start-up. For them this file offers one best
// response at caller-given prices that allocates nothing: the caller passes the table, the prices
// and the output buffers (all device memory it owns); the only scratch — the per-unit prices of
// every scenario — lives in a file-scope device array of fixed size that every GPU loading the
// library keeps until the process exits.
//
// The evaluation is the plain exact variant of the library's evaluation pass: one warp per job, every
// option's reduced cost s = fma(p_{R-1}, u_{R-1}, ... fma(p_0, u_0, -v)) in fp64, the lexicographic
// minimum of (s, local index), the chosen units added to the caller's demand array with 64-bit
// atomics. Results are identical to esp_evaluate on the same inputs.

#include <cmath>
#include <cstdint>
#include <mutex>

#include <cuda_runtime.h>

#include "esp.h"

namespace {

// Scratch: per-unit prices p = lambda (RAW) or lambda / C (NORMALIZED) of every scenario.
constexpr int kNoallocMaxPrices = 65536;   // S * R at most (512 KiB of fp64)
static __device__ __align__(256) double g_noalloc_prices[kNoallocMaxPrices];

constexpr int kMaxDevices = 64;
std::mutex g_setup_mutex;
double *g_prices_ptr[kMaxDevices] = {};

// Device address of the scratch array on the current device; looked up once per device (the host
// name of the array is only a stand-in and must never be passed to a kernel). The address is kept
// for the life of the process: after cudaDeviceReset (or any teardown of the device's primary
// context) it is stale, so the entry point must not be used across a device reset.
esp_status scratch_for_current_device(double **out)
{
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) {
        cudaGetLastError();
        return ESP_ERR_CUDA;
    }
    if (dev < 0 || dev >= kMaxDevices)
        return ESP_ERR_UNSUPPORTED;
    std::lock_guard<std::mutex> lock(g_setup_mutex);
    if (!g_prices_ptr[dev]) {
        void *p = nullptr;
        if (cudaGetSymbolAddress(&p, g_noalloc_prices) != cudaSuccess || p == nullptr) {
            cudaGetLastError();
            return ESP_ERR_CUDA;
        }
        g_prices_ptr[dev] = static_cast<double *>(p);
    }
    *out = g_prices_ptr[dev];
    return ESP_OK;
}

__global__ void k_noalloc_prices(int32_t S, int32_t R, const double *lambda, const int64_t *cap, int32_t mode,
                                 double *prices, unsigned long long *demand)
{
    const int64_t n = (int64_t)S * R;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x) {
        prices[i] = (mode == ESP_PRICE_NORMALIZED) ? lambda[i] / (double)cap[i] : lambda[i];
        demand[i] = 0ull;   // the demand output is accumulated with atomics below
    }
}

__global__ void k_noalloc_best_response(int32_t S, int32_t J, int32_t R, const int64_t *job_off,
                                        const int32_t *units, const double *values, const double *prices,
                                        int32_t *sel, unsigned long long *demand, double *min_score)
{
    const int lane = threadIdx.x & 31;
    const int64_t n_jobs = (int64_t)S * J;
    const int64_t warps = (int64_t)gridDim.x * (blockDim.x >> 5);
    for (int64_t j = (int64_t)blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5); j < n_jobs; j += warps) {
        const int64_t s = j / J;
        const int64_t a = job_off[j], b = job_off[j + 1];
        const double *p = prices + s * R;
        double best = INFINITY;
        long long best_i = 0x7fffffffffffffffLL;
        for (int64_t o = a + lane; o < b; o += 32) {
            double sc = -values[o];
            for (int r = 0; r < R; ++r)
                sc = __fma_rn(p[r], __int2double_rn(units[o * R + r]), sc);
            if (sc < best || (sc == best && o < best_i)) {
                best = sc;
                best_i = o;
            }
        }
        for (int d = 16; d >= 1; d >>= 1) {
            const double ob = __shfl_xor_sync(0xffffffffu, best, d);
            const long long oi = __shfl_xor_sync(0xffffffffu, best_i, d);
            if (ob < best || (ob == best && oi < best_i)) {
                best = ob;
                best_i = oi;
            }
        }
        if (lane == 0) {
            if (b <= a) {
                // an empty job chooses nothing, and no option of it is read
                sel[j] = -1;
                if (min_score)
                    min_score[j] = INFINITY;
            } else {
                sel[j] = (int32_t)(best_i - a);
                if (min_score)
                    min_score[j] = best;
                for (int r = 0; r < R; ++r)
                    atomicAdd(demand + s * R + r, (unsigned long long)(long long)units[best_i * R + r]);
            }
        }
    }
}

}  // namespace

extern "C" esp_status esp_evaluate_noalloc(int32_t S, int32_t J, int32_t R, const int64_t *job_offsets,
                                           const int32_t *units, const double *values, const int64_t *capacity,
                                           const double *lambda, int32_t mode, int32_t *sel, int64_t *demand,
                                           double *min_score, void *cuda_stream)
{
    if (S < 1 || J < 0 || R < 1 || R > 16 || !job_offsets || !capacity || !lambda || !sel || !demand ||
        (J > 0 && (!units || !values)))
        return ESP_ERR_INVALID_ARG;
    if (mode != ESP_PRICE_RAW && mode != ESP_PRICE_NORMALIZED)
        return ESP_ERR_INVALID_ARG;
    if ((int64_t)S * R > kNoallocMaxPrices)
        return ESP_ERR_INVALID_ARG;   // more prices than the fixed scratch array holds
    double *prices = nullptr;
    esp_status st = scratch_for_current_device(&prices);
    if (st != ESP_OK)
        return st;
    cudaStream_t stream = static_cast<cudaStream_t>(cuda_stream);
    unsigned long long *dem = reinterpret_cast<unsigned long long *>(demand);
    const int64_t n = (int64_t)S * R;
    k_noalloc_prices<<<(int)((n + 255) / 256), 256, 0, stream>>>(S, R, lambda, capacity, mode, prices, dem);
    if (cudaGetLastError() != cudaSuccess)
        return ESP_ERR_CUDA;
    const int64_t n_jobs = (int64_t)S * J;
    if (n_jobs > 0) {
        int64_t blocks = (n_jobs + 7) / 8;
        if (blocks > 65536)
            blocks = 65536;
        k_noalloc_best_response<<<(int)blocks, 256, 0, stream>>>(S, J, R, job_offsets, units, values, prices, sel,
                                                                  dem, min_score);
        if (cudaGetLastError() != cudaSuccess)
            return ESP_ERR_CUDA;
    }
    return ESP_OK;
}
