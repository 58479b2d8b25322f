// IAC slowdown predictor (include/esp_iac.h): the pair features of Sec. 3.4.1 and the three-layer
// network of Sec. 3.4.2 / Eq. dnn_pred, batched over co-location pairs.
//
// One thread per pair. The folded parameters (at most 64 hidden units: 6,593 fp32, 26 KB) travel
// as the kernel's own __grid_constant__ argument, which lives in the constant bank: with every loop
// unrolled each weight is a compile-time constant-bank operand of its fused multiply-add, so the
// two hidden layers are a straight run of FFMAs with no loads (no shared-memory staging, no global
// state shared between handles). The 14-float rows of the pair are gathered with 8-byte loads (the
// row table is small and stays in L2); the pair list and the output stream through once.

#include <cmath>
#include <cstdint>
#include <cstring>
#include <new>
#include <vector>

#include <cuda_runtime.h>

#include "esp_iac.h"

namespace {

constexpr int kFeat = ESP_IAC_FEATURES;   // 14
constexpr int kIn = ESP_IAC_INPUTS;       // 36
constexpr int kIacThreads = 256;

template <int H>
struct IacParams {
    float w1[H * kIn];   // row o: the 36 folded weights of hidden unit o
    float b1[H];
    float w2[H * H];
    float b2[H];
    float w3[H];
    float b3;
};
static_assert(sizeof(IacParams<64>) + 64 <= 32764, "kernel argument limit");

// DRAM Active per unit of SM Active; a row with SM Active 0 contributes 0.
__device__ __forceinline__ float intensity(float sm, float dram)
{
    return sm == 0.0f ? 0.0f : __fdiv_rn(dram, sm);
}

template <int H>
__global__ void __launch_bounds__(kIacThreads) k_iac(const __grid_constant__ IacParams<H> w, const float *jf,
                                                     int32_t n_rows, const int2 *pairs, int64_t n_pairs,
                                                     float c_mem, float *out)
{
    const int64_t stride = (int64_t)gridDim.x * kIacThreads;
    for (int64_t p = (int64_t)blockIdx.x * kIacThreads + threadIdx.x; p < n_pairs; p += stride) {
        const int2 ij = __ldg(pairs + p);
        if ((uint32_t)ij.x >= (uint32_t)n_rows || (uint32_t)ij.y >= (uint32_t)n_rows) {
            out[p] = __int_as_float(0x7fffffff);
            continue;
        }
        float x[kIn];
        const float2 *ra = reinterpret_cast<const float2 *>(jf + (size_t)ij.x * kFeat);
        const float2 *rb = reinterpret_cast<const float2 *>(jf + (size_t)ij.y * kFeat);
#pragma unroll
        for (int q = 0; q < kFeat / 2; ++q) {
            const float2 va = __ldg(ra + q), vb = __ldg(rb + q);
            x[2 * q] = va.x;
            x[2 * q + 1] = va.y;
            x[kFeat + 2 * q] = vb.x;
            x[kFeat + 2 * q + 1] = vb.y;
        }
        const float *a = x, *b = x + kFeat;
        // pairwise block: mean utilizations, co-location type, memory pressure, compute balance,
        // memory intensity difference
        x[28] = __fmul_rn(__fadd_rn(a[0], b[0]), 0.5f);
        x[29] = __fmul_rn(__fadd_rn(a[1], b[1]), 0.5f);
        x[30] = __fmul_rn(__fadd_rn(a[2], b[2]), 0.5f);
        x[31] = __fmul_rn(__fadd_rn(a[4], b[4]), 0.5f);
        x[32] = __fadd_rn(a[5], b[5]);
        x[33] = __fdiv_rn(__fadd_rn(a[3], b[3]), c_mem);
        const float lo = fminf(a[0], b[0]), hi = fmaxf(a[0], b[0]);
        x[34] = hi == 0.0f ? 1.0f : __fdiv_rn(lo, hi);
        x[35] = fabsf(__fsub_rn(intensity(a[0], a[2]), intensity(b[0], b[2])));

        float h1[H];
#pragma unroll
        for (int o = 0; o < H; ++o) {
            float acc = w.b1[o];
#pragma unroll
            for (int i = 0; i < kIn; ++i)
                acc = __fmaf_rn(w.w1[o * kIn + i], x[i], acc);
            h1[o] = fmaxf(acc, 0.0f);
        }
        float y = w.b3;
#pragma unroll
        for (int o = 0; o < H; ++o) {
            float acc = w.b2[o];
#pragma unroll
            for (int i = 0; i < H; ++i)
                acc = __fmaf_rn(w.w2[o * H + i], h1[i], acc);
            y = __fmaf_rn(w.w3[o], fmaxf(acc, 0.0f), y);
        }
        out[p] = __fadd_rn(1.0f, fmaxf(y, 0.0f));
    }
}

template <int H>
void fill_params(IacParams<H> &dst, int hp, const std::vector<float> &w1, const std::vector<float> &b1,
                 const std::vector<float> &w2, const std::vector<float> &b2, const std::vector<float> &w3, float b3)
{
    std::memset(&dst, 0, sizeof(dst));   // padded units: zero weights and biases, so they stay 0
    for (int o = 0; o < hp; ++o) {
        for (int i = 0; i < kIn; ++i)
            dst.w1[o * kIn + i] = w1[(size_t)o * kIn + i];
        dst.b1[o] = b1[o];
        for (int i = 0; i < hp; ++i)
            dst.w2[o * H + i] = w2[(size_t)o * hp + i];
        dst.b2[o] = b2[o];
        dst.w3[o] = w3[o];
    }
    dst.b3 = b3;
}

}  // namespace

struct esp_iac {
    int device = 0;
    int sm_count = 0;
    cudaStream_t stream = nullptr;
    bool loaded = false;
    bool poisoned = false;
    int H = 0;       // hidden units of the loaded model
    int Hk = 0;      // kernel width (16, 32 or 64; extra units are zero)
    IacParams<16> p16;
    IacParams<32> p32;
    IacParams<64> p64;
    int grid_cap = 0;
    int64_t launches = 0;
    // buffers of esp_iac_predict_host
    float *d_rows = nullptr, *d_out = nullptr;
    int2 *d_pairs = nullptr;
    size_t cap_rows = 0, cap_pairs = 0, cap_out = 0;
};

namespace {

esp_status fail(esp_iac *m, cudaError_t)
{
    cudaGetLastError();
    if (m)
        m->poisoned = true;
    return ESP_ERR_CUDA;
}

#define IAC_CUDA(call)                 \
    do {                               \
        cudaError_t e_ = (call);       \
        if (e_ != cudaSuccess)         \
            return fail(m, e_);        \
    } while (0)

esp_status check_handle(esp_iac *m)
{
    if (!m)
        return ESP_ERR_INVALID_ARG;
    if (m->poisoned)
        return ESP_ERR_STATE;
    return ESP_OK;
}

template <int H>
cudaError_t launch_iac(esp_iac *m, const IacParams<H> &w, int32_t n_rows, const float *rows, int64_t n_pairs,
                       const int2 *pairs, float c_mem, float *out)
{
    const int64_t blocks = (n_pairs + kIacThreads - 1) / kIacThreads;
    const int grid = (int)std::min<int64_t>(blocks, m->grid_cap);
    k_iac<H><<<grid, kIacThreads, 0, m->stream>>>(w, rows, n_rows, pairs, n_pairs, c_mem, out);
    return cudaGetLastError();
}

esp_status enqueue(esp_iac *m, int32_t n_rows, const float *rows, int64_t n_pairs, const int2 *pairs, float c_mem,
                   float *out)
{
    m->launches = 0;
    if (n_pairs == 0)
        return ESP_OK;
    IAC_CUDA(cudaSetDevice(m->device));
    cudaError_t e;
    if (m->Hk == 16)
        e = launch_iac<16>(m, m->p16, n_rows, rows, n_pairs, pairs, c_mem, out);
    else if (m->Hk == 32)
        e = launch_iac<32>(m, m->p32, n_rows, rows, n_pairs, pairs, c_mem, out);
    else
        e = launch_iac<64>(m, m->p64, n_rows, rows, n_pairs, pairs, c_mem, out);
    if (e != cudaSuccess)
        return fail(m, e);
    m->launches = 1;
    return ESP_OK;
}

bool finite_all(const float *p, size_t n)
{
    for (size_t i = 0; i < n; ++i)
        if (!std::isfinite(p[i]))
            return false;
    return true;
}

// BN folded into the layer: W' = s W, b' = s (b - mean) + beta, s = gamma / sqrt(var + eps), in fp64,
// rounded once to fp32. Returns false on a non-positive var + eps or a result beyond fp32.
bool fold(int H, int fan_in, const float *W, const float *b, const float *bn, double eps, std::vector<float> &Wf,
          std::vector<float> &bf)
{
    Wf.assign((size_t)H * fan_in, 0.0f);
    bf.assign((size_t)H, 0.0f);
    for (int o = 0; o < H; ++o) {
        const double gamma = bn[o], beta = bn[H + o], mean = bn[2 * H + o], var = bn[3 * H + o];
        const double d = var + eps;
        if (!(d > 0.0))
            return false;
        const double s = gamma / std::sqrt(d);
        for (int i = 0; i < fan_in; ++i) {
            const double v = s * (double)W[(size_t)o * fan_in + i];
            if (!(std::fabs(v) <= 3.4028234663852886e38))
                return false;
            Wf[(size_t)o * fan_in + i] = (float)v;
        }
        const double c = s * ((double)b[o] - mean) + beta;
        if (!(std::fabs(c) <= 3.4028234663852886e38))
            return false;
        bf[o] = (float)c;
    }
    return true;
}

template <typename T>
esp_status grow(esp_iac *m, T **p, size_t &cap, size_t count)
{
    if (count <= cap && *p)
        return ESP_OK;
    if (*p) {
        IAC_CUDA(cudaFree(*p));
        *p = nullptr;
        cap = 0;
    }
    void *q = nullptr;
    if (cudaMalloc(&q, std::max<size_t>(count, 1) * sizeof(T)) != cudaSuccess) {
        cudaGetLastError();
        return ESP_ERR_OOM;
    }
    *p = static_cast<T *>(q);
    cap = count;
    return ESP_OK;
}

}  // namespace

extern "C" {

esp_status esp_iac_create(esp_iac **out, int device, void *cuda_stream)
{
    if (!out)
        return ESP_ERR_INVALID_ARG;
    *out = nullptr;
    int n = 0;
    if (cudaGetDeviceCount(&n) != cudaSuccess || n == 0) {
        cudaGetLastError();
        return ESP_ERR_UNSUPPORTED;
    }
    if (device < 0 && cudaGetDevice(&device) != cudaSuccess)
        return ESP_ERR_CUDA;
    if (device >= n)
        return ESP_ERR_INVALID_ARG;
    cudaDeviceProp prop;
    if (cudaGetDeviceProperties(&prop, device) != cudaSuccess)
        return ESP_ERR_CUDA;
    if (prop.major != 10 || prop.minor != 3)
        return ESP_ERR_UNSUPPORTED;
    esp_iac *m = new (std::nothrow) esp_iac();
    if (!m)
        return ESP_ERR_OOM;
    m->device = device;
    m->stream = static_cast<cudaStream_t>(cuda_stream);
    m->sm_count = prop.multiProcessorCount;
    if (cudaSetDevice(device) != cudaSuccess) {
        delete m;
        return ESP_ERR_CUDA;
    }
    *out = m;
    return ESP_OK;
}

esp_status esp_iac_set_stream(esp_iac *m, void *cuda_stream)
{
    const esp_status st = check_handle(m);
    if (st != ESP_OK)
        return st;
    m->stream = static_cast<cudaStream_t>(cuda_stream);
    return ESP_OK;
}

esp_status esp_iac_load_model(esp_iac *m, int32_t H, const float *W1, const float *b1, const float *bn1,
                              const float *W2, const float *b2, const float *bn2, const float *W3, float b3,
                              float eps)
{
    esp_status st = check_handle(m);
    if (st != ESP_OK)
        return st;
    if (H < 1 || H > ESP_IAC_MAX_HIDDEN || !W1 || !b1 || !bn1 || !W2 || !b2 || !bn2 || !W3)
        return ESP_ERR_INVALID_ARG;
    if (!finite_all(W1, (size_t)H * kIn) || !finite_all(b1, H) || !finite_all(bn1, 4 * (size_t)H) ||
        !finite_all(W2, (size_t)H * H) || !finite_all(b2, H) || !finite_all(bn2, 4 * (size_t)H) ||
        !finite_all(W3, H) || !std::isfinite(b3) || !std::isfinite(eps) || eps < 0.0f)
        return ESP_ERR_INVALID_ARG;
    std::vector<float> w1f, b1f, w2f, b2f;
    if (!fold(H, kIn, W1, b1, bn1, eps, w1f, b1f) || !fold(H, H, W2, b2, bn2, eps, w2f, b2f))
        return ESP_ERR_INVALID_ARG;
    std::vector<float> w3(W3, W3 + H);
    m->loaded = false;
    m->H = H;
    m->Hk = H <= 16 ? 16 : (H <= 32 ? 32 : 64);
    if (m->Hk == 16)
        fill_params<16>(m->p16, H, w1f, b1f, w2f, b2f, w3, b3);
    else if (m->Hk == 32)
        fill_params<32>(m->p32, H, w1f, b1f, w2f, b2f, w3, b3);
    else
        fill_params<64>(m->p64, H, w1f, b1f, w2f, b2f, w3, b3);
    // a grid-stride loop over the pairs: enough resident blocks to fill every SM
    int per_sm = 0;
    cudaError_t e;
    if (m->Hk == 16)
        e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, k_iac<16>, kIacThreads, 0);
    else if (m->Hk == 32)
        e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, k_iac<32>, kIacThreads, 0);
    else
        e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, k_iac<64>, kIacThreads, 0);
    if (e != cudaSuccess)
        return fail(m, e);
    m->grid_cap = std::max(1, per_sm) * m->sm_count * 8;
    m->loaded = true;
    return ESP_OK;
}

esp_status esp_iac_predict(esp_iac *m, int32_t n_rows, const float *job_features, int64_t n_pairs,
                           const int32_t *pairs, float c_mem, float *s_hat)
{
    esp_status st = check_handle(m);
    if (st != ESP_OK)
        return st;
    if (!m->loaded)
        return ESP_ERR_NOT_LOADED;
    if (n_rows < 0 || n_pairs < 0 || !(c_mem > 0.0f) || !std::isfinite(c_mem))
        return ESP_ERR_INVALID_ARG;
    if (n_pairs > 0 && (!pairs || !s_hat || (n_rows > 0 && !job_features)))
        return ESP_ERR_INVALID_ARG;
    if ((reinterpret_cast<uintptr_t>(job_features) & 7u) || (reinterpret_cast<uintptr_t>(pairs) & 7u))
        return ESP_ERR_INVALID_ARG;
    return enqueue(m, n_rows, job_features, n_pairs, reinterpret_cast<const int2 *>(pairs), c_mem, s_hat);
}

esp_status esp_iac_predict_host(esp_iac *m, int32_t n_rows, const float *job_features, int64_t n_pairs,
                                const int32_t *pairs, float c_mem, float *s_hat)
{
    esp_status st = check_handle(m);
    if (st != ESP_OK)
        return st;
    if (!m->loaded)
        return ESP_ERR_NOT_LOADED;
    if (n_rows < 0 || n_pairs < 0 || !(c_mem > 0.0f) || !std::isfinite(c_mem))
        return ESP_ERR_INVALID_ARG;
    if (n_pairs == 0) {
        m->launches = 0;
        return ESP_OK;
    }
    if (!pairs || !s_hat || (n_rows > 0 && !job_features))
        return ESP_ERR_INVALID_ARG;
    for (int64_t q = 0; q < 2 * n_pairs; ++q)
        if (pairs[q] < 0 || pairs[q] >= n_rows)
            return ESP_ERR_INVALID_ARG;
    IAC_CUDA(cudaSetDevice(m->device));
    if ((st = grow(m, &m->d_rows, m->cap_rows, (size_t)n_rows * kFeat)) != ESP_OK)
        return st;
    if ((st = grow(m, &m->d_pairs, m->cap_pairs, (size_t)n_pairs)) != ESP_OK)
        return st;
    if ((st = grow(m, &m->d_out, m->cap_out, (size_t)n_pairs)) != ESP_OK)
        return st;
    IAC_CUDA(cudaMemcpyAsync(m->d_rows, job_features, (size_t)n_rows * kFeat * sizeof(float), cudaMemcpyHostToDevice,
                             m->stream));
    IAC_CUDA(cudaMemcpyAsync(m->d_pairs, pairs, (size_t)n_pairs * sizeof(int2), cudaMemcpyHostToDevice, m->stream));
    if ((st = enqueue(m, n_rows, m->d_rows, n_pairs, m->d_pairs, c_mem, m->d_out)) != ESP_OK)
        return st;
    IAC_CUDA(cudaMemcpyAsync(s_hat, m->d_out, (size_t)n_pairs * sizeof(float), cudaMemcpyDeviceToHost, m->stream));
    IAC_CUDA(cudaStreamSynchronize(m->stream));
    return ESP_OK;
}

esp_status esp_iac_last_launch_count(esp_iac *m, int64_t *out)
{
    if (!m || !out)
        return ESP_ERR_INVALID_ARG;
    *out = m->launches;
    return ESP_OK;
}

void esp_iac_destroy(esp_iac *m)
{
    if (!m)
        return;
    cudaSetDevice(m->device);
    if (m->d_rows)
        cudaFree(m->d_rows);
    if (m->d_pairs)
        cudaFree(m->d_pairs);
    if (m->d_out)
        cudaFree(m->d_out);
    cudaGetLastError();
    delete m;
}

}  // extern "C"
