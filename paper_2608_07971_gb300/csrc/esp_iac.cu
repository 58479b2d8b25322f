// IAC slowdown predictor (include/esp_iac.h): the pair features of Sec. 3.3.1 and the three-layer
// network of Sec. 3.3.2 / Eq. dnn_pred, batched over co-location pairs.
//
// Two kernels compute it. k_iac_tc (the default) runs the hidden layers on the tensor cores
// (esp_iac_tc.cuh). k_iac is the CUDA-core kernel: one thread per pair. The folded parameters (at most 64 hidden units: 6,593 fp32, 26 KB) travel
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

#include "esp_debug.h"
#include "esp_iac.h"
#include "esp_iac_tc.cuh"

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


// ---- tensor-core path (esp_iac_tc.cuh)

static_assert(kIn < iac_tc::kK1, "X has a padding column for layer 1's bias");

struct IacEpilogue {
    float b2[iac_tc::kN];   // folded layer-2 bias (zero beyond H); layer 1's enters the MMAs
    float w3[iac_tc::kN];
    float b3;
};

constexpr uint32_t kIacWaitSuspendNs = 1000000;
constexpr uint32_t kIacWaitPolls = 4096;     // about 4 s of waiting before a timeout is reported
constexpr unsigned int kIacErrTimeout = 1u;

__device__ __forceinline__ uint32_t smem_addr(const void *p)
{
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

// Shared-memory matrix descriptor: start address, leading and stride byte offsets (16-byte units),
// descriptor version 1 (bits 46-47), no swizzle (bits 61-63 = 0).
__device__ __forceinline__ uint64_t smem_desc(uint32_t addr, uint32_t lbo, uint32_t sbo)
{
    return (uint64_t)((addr >> 4) & 0x3fffu) | ((uint64_t)((lbo >> 4) & 0x3fffu) << 16) |
           ((uint64_t)((sbo >> 4) & 0x3fffu) << 32) | (1ull << 46);
}

__device__ __forceinline__ void mma_tf32(uint32_t d_tmem, uint64_t a, uint64_t b, uint32_t accumulate)
{
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "setp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::tf32 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
        "l"(a), "l"(b), "r"(iac_tc::kIdesc), "r"(accumulate)
        : "memory");
}

// The same MMA with A in tensor memory (lane = row, one tf32 column per k), B from shared memory.
__device__ __forceinline__ void mma_tf32_ts(uint32_t d_tmem, uint32_t a_tmem, uint64_t b, uint32_t accumulate)
{
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "setp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::tf32 [%0], [%1], %2, %3, p;\n\t}" ::"r"(d_tmem),
        "r"(a_tmem), "l"(b), "r"(iac_tc::kIdesc), "r"(accumulate)
        : "memory");
}

__device__ __forceinline__ void mma_commit(uint32_t bar)
{
    asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar)
                 : "memory");
}

__device__ __forceinline__ void tc_fence_before()
{
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}

__device__ __forceinline__ void tc_fence_after()
{
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}

__device__ __forceinline__ void fence_async_smem()
{
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

// Barrier of one warpgroup (named barrier id, 128 threads) that also ANDs a predicate over it.
__device__ __forceinline__ bool wg_sync_and(int id, bool v)
{
    uint32_t r;
    asm volatile(
        "{\n\t.reg .pred p, q;\n\t"
        "setp.ne.b32 p, %1, 0;\n\t"
        "bar.red.and.pred q, %2, 128, p;\n\t"
        "selp.u32 %0, 1, 0, q;\n\t}"
        : "=r"(r)
        : "r"((uint32_t)v), "r"(id)
        : "memory");
    return r != 0;
}

__device__ __forceinline__ bool mbar_wait_bounded(uint32_t bar, uint32_t parity, uint32_t polls)
{
    for (uint32_t it = 0; it < polls; ++it) {
        uint32_t done;
        asm volatile(
            "{\n\t.reg .pred p;\n\t"
            "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2, %3;\n\t"
            "selp.u32 %0, 1, 0, p;\n\t}"
            : "=r"(done)
            : "r"(bar), "r"(parity), "r"(kIacWaitSuspendNs)
            : "memory");
        if (done)
            return true;
    }
    return false;
}

// 32 consecutive fp32 columns of this thread's TMEM lane.
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, float *v)
{
    uint32_t r[32];
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, "
        "%15, %16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31}, [%32];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
          "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]),
          "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]),
          "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
        : "r"(taddr)
        : "memory");
#pragma unroll
    for (int i = 0; i < 32; ++i)
        v[i] = __uint_as_float(r[i]);
}

__device__ __forceinline__ void tmem_wait_ld()
{
    asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
}

// 32 consecutive 32-bit columns of this thread's TMEM lane.
__device__ __forceinline__ void tmem_st32(uint32_t taddr, const uint32_t *r)
{
    asm volatile(
        "tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], {%1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, "
        "%15, %16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31, %32};" ::"r"(taddr),
        "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]), "r"(r[8]),
        "r"(r[9]), "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]), "r"(r[15]), "r"(r[16]),
        "r"(r[17]), "r"(r[18]), "r"(r[19]), "r"(r[20]), "r"(r[21]), "r"(r[22]), "r"(r[23]), "r"(r[24]),
        "r"(r[25]), "r"(r[26]), "r"(r[27]), "r"(r[28]), "r"(r[29]), "r"(r[30]), "r"(r[31])
        : "memory");
}

__device__ __forceinline__ void tmem_wait_st()
{
    asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
}

// 32 values split into tf32 high and low parts.
__device__ __forceinline__ void split32(const float *h, uint32_t *hi, uint32_t *lo)
{
    using namespace iac_tc;
#pragma unroll
    for (int i = 0; i < 32; ++i) {
        hi[i] = tf32_trunc_bits(__float_as_uint(h[i]));
        lo[i] = tf32_round_bits(__float_as_uint(__fsub_rn(h[i], __uint_as_float(hi[i]))));
    }
}

// Four consecutive values of a row, split into tf32 high and low parts, stored as one 16-byte chunk
// of each part.
__device__ __forceinline__ void store_split4(unsigned char *hi, unsigned char *lo, int off, float a, float b, float c,
                                             float d)
{
    using namespace iac_tc;
    const uint32_t ha = tf32_trunc_bits(__float_as_uint(a)), hb = tf32_trunc_bits(__float_as_uint(b));
    const uint32_t hc = tf32_trunc_bits(__float_as_uint(c)), hd = tf32_trunc_bits(__float_as_uint(d));
    const uint32_t la = tf32_round_bits(__float_as_uint(__fsub_rn(a, __uint_as_float(ha))));
    const uint32_t lb = tf32_round_bits(__float_as_uint(__fsub_rn(b, __uint_as_float(hb))));
    const uint32_t lc = tf32_round_bits(__float_as_uint(__fsub_rn(c, __uint_as_float(hc))));
    const uint32_t ld = tf32_round_bits(__float_as_uint(__fsub_rn(d, __uint_as_float(hd))));
    *reinterpret_cast<uint4 *>(hi + off) = make_uint4(ha, hb, hc, hd);
    *reinterpret_cast<uint4 *>(lo + off) = make_uint4(la, lb, lc, ld);
}

// A pair's two feature rows (zero when the pair is past the end or out of range).
struct PairRows {
    float2 a[kFeat / 2], b[kFeat / 2];
    bool valid;
};

__device__ __forceinline__ void fetch_pair(PairRows &r, int64_t p, int64_t n_pairs, const int2 *pairs,
                                           const float *jf, int32_t n_rows)
{
#pragma unroll
    for (int q = 0; q < kFeat / 2; ++q)
        r.a[q] = r.b[q] = make_float2(0.0f, 0.0f);
    r.valid = false;
    if (p < n_pairs) {
        const int2 ij = __ldg(pairs + p);
        r.valid = (uint32_t)ij.x < (uint32_t)n_rows && (uint32_t)ij.y < (uint32_t)n_rows;
        if (r.valid) {
            const float2 *ra = reinterpret_cast<const float2 *>(jf + (size_t)ij.x * kFeat);
            const float2 *rb = reinterpret_cast<const float2 *>(jf + (size_t)ij.y * kFeat);
#pragma unroll
            for (int q = 0; q < kFeat / 2; ++q) {
                r.a[q] = __ldg(ra + q);
                r.b[q] = __ldg(rb + q);
            }
        }
    }
}

// Issues the MMAs of one operand slice (three split products per k-step, ks_n k-steps): A from the
// warpgroup's buffer (hi, lo) with row-group stride a_sbo, B from the staged weights at b_hi / b_lo
// (k-step b_ks0 onwards, row-group stride b_sbo). acc0: the first product accumulates into D.
__device__ __forceinline__ void issue_split_mmas(uint32_t d, uint32_t a_hi, uint32_t a_lo, uint32_t a_sbo,
                                                 uint32_t b_hi, uint32_t b_lo, uint32_t b_sbo, int b_ks0, int ks_n,
                                                 bool acc0)
{
    for (int ks = 0; ks < ks_n; ++ks) {
        const uint64_t ah = smem_desc(a_hi + ks * 256, 128, a_sbo);
        const uint64_t al = smem_desc(a_lo + ks * 256, 128, a_sbo);
        const uint64_t bh = smem_desc(b_hi + (b_ks0 + ks) * 256, 128, b_sbo);
        const uint64_t bl = smem_desc(b_lo + (b_ks0 + ks) * 256, 128, b_sbo);
        mma_tf32(d, ah, bh, (acc0 || ks > 0) ? 1u : 0u);
        mma_tf32(d, ah, bl, 1u);
        mma_tf32(d, al, bh, 1u);
    }
}

// Layer 2's MMAs for one half of H1 (ks_n k-steps): A from tensor memory (hi at a_t, lo at
// a_t + 32), B from the staged weights at b_hi / b_lo (k-step b_ks0 onwards, row-group stride b_sbo).
__device__ __forceinline__ void issue_split_mmas_ts(uint32_t d, uint32_t a_t, uint32_t b_hi, uint32_t b_lo,
                                                    uint32_t b_sbo, int b_ks0, int ks_n, bool acc0)
{
    for (int ks = 0; ks < ks_n; ++ks) {
        const uint32_t ah = a_t + 8 * ks, al = a_t + iac_tc::kKH + 8 * ks;
        const uint64_t bh = smem_desc(b_hi + (b_ks0 + ks) * 256, 128, b_sbo);
        const uint64_t bl = smem_desc(b_lo + (b_ks0 + ks) * 256, 128, b_sbo);
        mma_tf32_ts(d, ah, bh, (acc0 || ks > 0) ? 1u : 0u);
        mma_tf32_ts(d, ah, bl, 1u);
        mma_tf32_ts(d, al, bh, 1u);
    }
}

// wait_polls: bounded waits poll this many times (a suspend of up to 1 ms each); hold != 0 (a
// failure-detection hook): the first MMA group of CTA 0's first warpgroup is never committed, so that
// warpgroup's wait runs out.
__global__ void __launch_bounds__(iac_tc::kThreads, 1) k_iac_tc(const __grid_constant__ IacEpilogue ep,
                                                                 const uint4 *bimg, const float *jf, int32_t n_rows,
                                                                 const int2 *pairs, int64_t n_pairs, float c_mem,
                                                                 float *out, unsigned int *err, uint32_t wait_polls,
                                                                 int32_t hold)
{
    using namespace iac_tc;
    extern __shared__ unsigned char smem_raw[];
    unsigned char *sm = reinterpret_cast<unsigned char *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                                          ~static_cast<uintptr_t>(1023));
    const int tid = threadIdx.x, wg = tid >> 7, row = tid & 127, warp = tid >> 5;
    uint64_t *bars = reinterpret_cast<uint64_t *>(sm + kOffBar);
    uint32_t *slot = reinterpret_cast<uint32_t *>(sm + kOffSlot);

    // the split weights, once per CTA
    for (int i = tid; i < kBImgBytes / 16; i += kThreads)
        reinterpret_cast<uint4 *>(sm)[i] = __ldg(bimg + i);
    if (tid == 0) {
        for (int g = 0; g < kWG; ++g)
            asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;" ::"r"(smem_addr(bars + g)) : "memory");
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    if (warp == 0) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_addr(slot)),
                     "r"(kTmemCols)
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
    fence_async_smem();
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *slot;
    const uint32_t lane_sel = (uint32_t)(32 * (warp & 3)) << 16;   // this warp's quarter of the lanes
    // the warpgroup's two regions of 64 columns: a tile's accumulators (D1, then D2) in one, its half
    // of H1 in the other, the roles swapped from one tile to the next
    const uint32_t t_base = tmem + (uint32_t)(wg * 2 * kN);
    unsigned char *a_hi = sm + kOffA + wg * kABufBytes, *a_lo = a_hi + kA1Bytes;
    const uint32_t a_hi_s = smem_addr(a_hi), a_lo_s = smem_addr(a_lo), sm_s = smem_addr(sm);
    const uint32_t bar = smem_addr(bars + wg);
    const int bar_id = 1 + wg;
    // the thread that issues the warpgroup's MMAs: lane 0 of its warp wg, so that the four issuers
    // sit in four different SM sub-partitions (warp w runs on sub-partition w mod 4)
    const bool issuer = row == 32 * wg;
    uint32_t phase = 0;
    bool ok = true;
    // The MMA groups are committed to the warpgroup's mbarrier one at a time. Every thread waits for
    // a group itself (bounded), agreed warp-wide so that the warp-collective tcgen05 loads and stores
    // after it run in every lane or in none; the warpgroup-wide agreement is taken at the next
    // hand-off barrier, which a timeout in any warp turns into a common exit.
    auto wait_group = [&]() {
        const bool mine = mbar_wait_bounded(bar, phase, wait_polls);
        phase ^= 1u;
        return __all_sync(0xffffffffu, mine);
    };
    // Hands the warpgroup's operand writes (X in shared memory, H1 in tensor memory) to the MMA issuer
    // and ANDs the waits of every warp; false: some warp's wait ran out.
    auto hand_off = [&](bool mine) {
        fence_async_smem();
        tc_fence_before();
        ok = wg_sync_and(bar_id, mine);
        tc_fence_after();
        return ok;
    };
    // a pair's 36 inputs (Sec. 3.3.1), zero for a pair past the end or out of range, split into X
    auto store_inputs = [&](const PairRows &r) {
        float x[kK1];
#pragma unroll
        for (int q = 0; q < kFeat / 2; ++q) {
            x[2 * q] = r.a[q].x;
            x[2 * q + 1] = r.a[q].y;
            x[kFeat + 2 * q] = r.b[q].x;
            x[kFeat + 2 * q + 1] = r.b[q].y;
        }
        x[kIn] = 1.0f;   // the column that carries layer 1's bias
#pragma unroll
        for (int i = kIn + 1; i < kK1; ++i)
            x[i] = 0.0f;
        if (r.valid) {
            const float *a = x, *b = x + kFeat;
            x[28] = __fmul_rn(__fadd_rn(a[0], b[0]), 0.5f);
            x[29] = __fmul_rn(__fadd_rn(a[1], b[1]), 0.5f);
            x[30] = __fmul_rn(__fadd_rn(a[2], b[2]), 0.5f);
            x[31] = __fmul_rn(__fadd_rn(a[4], b[4]), 0.5f);
            x[32] = __fadd_rn(a[5], b[5]);
            x[33] = __fdiv_rn(__fadd_rn(a[3], b[3]), c_mem);
            const float lo = fminf(a[0], b[0]), hi = fmaxf(a[0], b[0]);
            x[34] = hi == 0.0f ? 1.0f : __fdiv_rn(lo, hi);
            x[35] = fabsf(__fsub_rn(intensity(a[0], a[2]), intensity(b[0], b[2])));
        }
#pragma unroll
        for (int c = 0; c < kK1 / 4; ++c)
            store_split4(a_hi, a_lo, cm_off(row, 4 * c, kK1), x[4 * c], x[4 * c + 1], x[4 * c + 2], x[4 * c + 3]);
    };
    // layer 1 of a tile: D1 = X W1'^T into region d (hold: this group is not committed), after a
    // hand-off of the tile's X
    auto issue_layer1 = [&](uint32_t d, bool hold_group) {
        if (issuer) {
            issue_split_mmas(d, a_hi_s, a_lo_s, kK1 / 4 * 128, sm_s + kOffB1Hi, sm_s + kOffB1Lo, kK1 / 4 * 128, 0,
                             kK1 / 8, false);
            if (!hold_group)
                mma_commit(bar);
        }
        __syncwarp();
    };

    const int64_t tile_stride = (int64_t)gridDim.x * kWG;
    int64_t tile = (int64_t)blockIdx.x * kWG + wg;
    uint32_t par = 0;   // region of the current tile's accumulators
    bool valid = false;
    if (tile * kM < n_pairs) {
        PairRows first;
        fetch_pair(first, tile * kM + row, n_pairs, pairs, jf, n_rows);
        store_inputs(first);
        valid = first.valid;
        hand_off(true);
        issue_layer1(t_base, hold != 0 && blockIdx.x == 0 && wg == 0);
    }
    for (; tile * kM < n_pairs; tile += tile_stride, par ^= 1u) {
        const int64_t p = tile * kM + row;
        const uint32_t tD = t_base + par * kN, tH = t_base + (par ^ 1u) * kN;   // MMA view (lane 0)
        const uint32_t tD_w = tD | lane_sel, tH_w = tH | lane_sel;             // this warp's lanes
        const bool more = (tile + tile_stride) * kM < n_pairs;
        // ---- epilogue 1: h1 = ReLU(D1) (D1 holds the bias); the first half split into H, the second kept in
        // registers
        bool mine = wait_group();   // layer 1
        float h[32];
        if (mine) {
            tc_fence_after();
            float v[64];
            tmem_ld32(tD_w, v);
            tmem_ld32(tD_w + kKH, v + kKH);
            tmem_wait_ld();
            uint32_t hi[32], lo[32];
#pragma unroll
            for (int i = 0; i < 32; ++i)
                h[i] = fmaxf(v[i], 0.0f);
            split32(h, hi, lo);
            tmem_st32(tH_w, hi);
            tmem_st32(tH_w + kKH, lo);
#pragma unroll
            for (int i = 0; i < 32; ++i)
                h[i] = fmaxf(v[kKH + i], 0.0f);
            tmem_wait_st();
        }
        if (!hand_off(mine))   // D1 is read (its region takes D2), the first half of H1 is in H
            break;
        // ---- layer 2, first half: D2 = H1[:, 0..31] W2'[:, 0..31]^T
        if (issuer) {
            issue_split_mmas_ts(tD, tH, sm_s + kOffB2Hi, sm_s + kOffB2Lo, kK2 / 4 * 128, 0, kKH / 8, false);
            mma_commit(bar);
        }
        __syncwarp();
        // while those MMAs run: the second half's split, and the next tile's pair and rows
        uint32_t hi2[32], lo2[32];
        split32(h, hi2, lo2);
        PairRows nxt;
        fetch_pair(nxt, p + tile_stride * kM, n_pairs, pairs, jf, n_rows);
        mine = wait_group();   // the first half's MMAs have read H
        if (mine) {
            tc_fence_after();
            tmem_st32(tH_w, hi2);
            tmem_st32(tH_w + kKH, lo2);
            tmem_wait_st();
        }
        if (!hand_off(mine))
            break;
        // ---- layer 2, second half: D2 += H1[:, 32..63] W2'[:, 32..63]^T
        if (issuer) {
            issue_split_mmas_ts(tD, tH, sm_s + kOffB2Hi, sm_s + kOffB2Lo, kK2 / 4 * 128, kKH / 8, kKH / 8, true);
            mma_commit(bar);
        }
        __syncwarp();
        // the next tile's inputs while those MMAs run (the MMAs that read X have completed)
        const bool cur_valid = valid;
        if (more) {
            store_inputs(nxt);
            valid = nxt.valid;
        }
        if (!hand_off(wait_group()))   // layer 2 is done; the next tile's X is in the buffer
            break;
        // the next tile's layer 1 into H (read by the MMAs just completed) runs during epilogue 2
        if (more)
            issue_layer1(tH, false);

        // ---- epilogue 2: S_hat = 1 + ReLU(b3 + sum_o w3_o ReLU(D2_o + b2'_o)), o in order
        float y = ep.b3;
        {
            float v[64];
            tmem_ld32(tD_w, v);
            tmem_ld32(tD_w + 32, v + 32);
            tmem_wait_ld();
#pragma unroll
            for (int o = 0; o < 64; ++o)
                y = __fmaf_rn(ep.w3[o], fmaxf(__fadd_rn(v[o], ep.b2[o]), 0.0f), y);
        }
        if (p < n_pairs)
            out[p] = cur_valid ? __fadd_rn(1.0f, fmaxf(y, 0.0f)) : __int_as_float(0x7fffffff);
        // the next tile's epilogue 1 writes this region (its half of H1) after these reads completed
    }
    if (!ok) {
        // an MMA group did not complete in time: the mbarrier is made to track every MMA of this
        // warpgroup still in flight, whose completion is awaited (bounded) before the tensor memory
        // is released; the timeout is reported
        if (issuer)
            mma_commit(bar);
        phase ^= 1u;   // the phase the failed wait was for
        mbar_wait_bounded(bar, phase, wait_polls);
        if (row == 0)
            atomicOr(err, kIacErrTimeout);
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (warp == 0)
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kTmemCols) : "memory");
}

// Split images of [W1' | b1'] (64 x 40: the bias in column 36, which meets X's column of ones) and W2'
// (64 x 64) in the canonical layout, hi then lo of each.
void build_bimg(int H, const std::vector<float> &w1, const std::vector<float> &b1, const std::vector<float> &w2,
                std::vector<uint32_t> &img)
{
    using namespace iac_tc;
    img.assign(kBImgBytes / 4, 0u);
    auto put = [&](int base, int K, int o, int k, float v) {
        uint32_t bits;
        std::memcpy(&bits, &v, 4);
        const uint32_t hi = tf32_trunc_bits(bits);
        float hf;
        std::memcpy(&hf, &hi, 4);
        const float lo = v - hf;   // exact: the bits below the tf32 mantissa
        uint32_t lb;
        std::memcpy(&lb, &lo, 4);
        const int B = (base == 0) ? kB1Bytes : kB2Bytes;
        img[(base + cm_off(o, k, K)) / 4] = hi;
        img[(base + B + cm_off(o, k, K)) / 4] = tf32_round_bits(lb);
    };
    for (int o = 0; o < H; ++o) {
        for (int k = 0; k < kIn; ++k)
            put(kOffB1Hi, kK1, o, k, w1[(size_t)o * kIn + k]);
        put(kOffB1Hi, kK1, o, kIn, b1[o]);
        for (int i = 0; i < H; ++i)
            put(kOffB2Hi, kK2, o, i, w2[(size_t)o * H + i]);
    }
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
    int path = ESP_IAC_PATH_TENSOR;
    IacEpilogue ep;                       // tensor path: biases and output weights
    std::vector<uint32_t> h_bimg;         // tensor path: split W1', W2' (host copy of the upload)
    uint4 *d_bimg = nullptr;
    unsigned int *d_err = nullptr;        // device error word (timeouts of the tensor path)
    // failure-detection hooks (esp_debug.h): polls of a bounded wait (about 1 ms each), and the next
    // tensor-path launch leaving one MMA group uncommitted
    uint32_t wait_polls = kIacWaitPolls;
    bool hold_commit = false;
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

cudaError_t launch_iac_tc(esp_iac *m, int32_t n_rows, const float *rows, int64_t n_pairs, const int2 *pairs,
                         float c_mem, float *out)
{
    const int64_t tiles = (n_pairs + iac_tc::kM - 1) / iac_tc::kM;
    const int grid = (int)std::min<int64_t>((tiles + iac_tc::kWG - 1) / iac_tc::kWG, m->sm_count);
    const int32_t hold = m->hold_commit ? 1 : 0;
    m->hold_commit = false;   // the hook holds one launch only
    k_iac_tc<<<grid, iac_tc::kThreads, iac_tc::kSmemBytes, m->stream>>>(m->ep, m->d_bimg, rows, n_rows, pairs,
                                                                       n_pairs, c_mem, out, m->d_err, m->wait_polls,
                                                                       hold);
    return cudaGetLastError();
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
    if (m->path == ESP_IAC_PATH_TENSOR)
        e = launch_iac_tc(m, n_rows, rows, n_pairs, pairs, c_mem, out);
    else if (m->Hk == 16)
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
    void *e = nullptr, *b = nullptr;
    if (cudaMalloc(&e, sizeof(unsigned int)) != cudaSuccess || cudaMalloc(&b, iac_tc::kBImgBytes) != cudaSuccess ||
        cudaMemset(e, 0, sizeof(unsigned int)) != cudaSuccess ||
        cudaFuncSetAttribute(k_iac_tc, cudaFuncAttributeMaxDynamicSharedMemorySize, iac_tc::kSmemBytes) !=
            cudaSuccess) {
        cudaGetLastError();
        if (e)
            cudaFree(e);
        if (b)
            cudaFree(b);
        delete m;
        return ESP_ERR_CUDA;
    }
    m->d_err = static_cast<unsigned int *>(e);
    m->d_bimg = static_cast<uint4 *>(b);
    *out = m;
    return ESP_OK;
}

esp_status esp_iac_set_path(esp_iac *m, int32_t path)
{
    const esp_status st = check_handle(m);
    if (st != ESP_OK)
        return st;
    if (path != ESP_IAC_PATH_TENSOR && path != ESP_IAC_PATH_FMA)
        return ESP_ERR_INVALID_ARG;
    m->path = path;
    return ESP_OK;
}

esp_status esp_iac_synchronize(esp_iac *m)
{
    const esp_status st = check_handle(m);
    if (st != ESP_OK)
        return st;
    IAC_CUDA(cudaSetDevice(m->device));
    IAC_CUDA(cudaStreamSynchronize(m->stream));
    unsigned int err = 0;
    IAC_CUDA(cudaMemcpy(&err, m->d_err, sizeof(err), cudaMemcpyDeviceToHost));
    if (err) {
        m->poisoned = true;
        return ESP_ERR_TIMEOUT;
    }
    return ESP_OK;
}

esp_status esp_iac_debug_set_wait_limit(esp_iac *m, uint32_t limit_ms)
{
    const esp_status st = check_handle(m);
    if (st != ESP_OK)
        return st;
    m->wait_polls = limit_ms == 0 ? kIacWaitPolls : limit_ms;
    return ESP_OK;
}

esp_status esp_iac_debug_hold_commit(esp_iac *m)
{
    const esp_status st = check_handle(m);
    if (st != ESP_OK)
        return st;
    if (m->path != ESP_IAC_PATH_TENSOR)
        return ESP_ERR_UNSUPPORTED;
    m->hold_commit = true;
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
    // tensor path: layer 2's bias and the output weights for the epilogue, split weight images (with
    // layer 1's bias) for the MMAs
    std::memset(&m->ep, 0, sizeof(m->ep));
    for (int o = 0; o < H; ++o) {
        m->ep.b2[o] = b2f[o];
        m->ep.w3[o] = w3[o];
    }
    m->ep.b3 = b3;
    build_bimg(H, w1f, b1f, w2f, m->h_bimg);
    IAC_CUDA(cudaSetDevice(m->device));
    IAC_CUDA(cudaMemcpyAsync(m->d_bimg, m->h_bimg.data(), iac_tc::kBImgBytes, cudaMemcpyHostToDevice, m->stream));
    IAC_CUDA(cudaStreamSynchronize(m->stream));
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
    return esp_iac_synchronize(m);
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
    if (m->d_bimg)
        cudaFree(m->d_bimg);
    if (m->d_err)
        cudaFree(m->d_err);
    cudaGetLastError();
    delete m;
}

}  // extern "C"
