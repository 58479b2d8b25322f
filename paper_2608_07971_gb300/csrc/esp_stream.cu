// Streaming evaluation pass of the ESP tatonnement (Sec. 3.2.2: every job's best response to the
// round's prices, Eq. esp_score without Gamma; the int64 demand of the choices; Eq. price_update
// fused into the pass) for sm_103a, for tables whose jobs all belong to runs of equal size (uniform
// tables, and the sorted layout of ragged tables whose jobs have at most 256 options).
//
// One persistent CTA per SM streams a static, contiguous range of blocks; a block is whole jobs of
// one run and scenario, at most a stage's options, described by one TileDesc. Per CTA
// kStreamProducers producer warps fill a ring of shared-memory stages, one block per stage: the
// block's descriptor by ordinary shared stores, its unit rows and values by two 1-D bulk copies
// (cp.async.bulk, the TMA engine) counted in on the stage's full barrier (expect_tx / complete_tx).
// Producer p issues the blocks p, p + P, p + 2P, ... (issuing a bulk copy costs its thread a few
// hundred cycles, so several warps issue in parallel). Each of kStreamConsumers consumer warps takes
// the CTA's next block (a shared counter), waits for its stage, evaluates it (the fp32 screen with
// its exact fp64 resolution, esp_tile.cuh: rows of 32 lanes x 4 options, or 2 x 4 options per lane
// for jobs of 132..256 options) and releases the stage alone (empty barrier of count 1): a slow warp
// holds one stage, not the ring, and no consumer issues a copy. The arithmetic per option and per job
// is the per-warp pass's (k_pass): selections, demands and prices are identical bit for bit.
//
// The price update: a consumer warp's demand stays in registers while it evaluates one scenario
// and is added to the scenario's int64 accumulator when the warp moves on, together with the number
// of the scenario's blocks it evaluated; the addition that completes the scenario's block count makes
// that warp apply Eq. price_update to it, after it has released the stage it holds.
//
// Every wait is bounded (SolveArgs::wait_ms of the GPU's global timer): on expiry the kernel flags
// DEV_ERR_TIMEOUT, one thread waits (bounded) for the copies still in flight, and the CTA returns.

#include <cmath>
#include <cstdint>
#include <cuda_runtime.h>

#include "esp_device.cuh"
#include "esp_kernels.h"
#include "esp_ptx.cuh"
#include "esp_tile.cuh"
#include "esp_warp.cuh"

namespace esp {

namespace {

// Issues block d, the CTA's block `index`, into a stage (one producer lane): its descriptor and then
// its index (the stage's sequence word) by shared stores, its units and values by two bulk copies
// widened to 16-byte boundaries, counted on the stage's full barrier. The
// stage's previous contents were read by its consumer before it arrived on the empty barrier the
// producer waited for, so neither the stores nor the copies overtake those reads.
__device__ __forceinline__ void issue_block(const DevTable &t, const int4 &dlo, const int4 &dhi, int index,
                                            unsigned char *stage, const StreamStageLayout &SL, uint32_t full,
                                            uint32_t extra_tx)
{
    const int R = t.R;
    const int64_t opt = (int64_t)(((uint64_t)(uint32_t)dlo.y << 32) | (uint32_t)dlo.x);
    const int n_opt = dhi.x;
    const int64_t ub = opt * R * 4, ue = (opt + n_opt) * R * 4;
    const int64_t ulo = ub & ~int64_t(15), uhi = (ue + 15) & ~int64_t(15);
    const int64_t vb = opt * 8, ve = (opt + n_opt) * 8;
    const int64_t vlo = vb & ~int64_t(15), vhi = (ve + 15) & ~int64_t(15);
    reinterpret_cast<int4 *>(stage + SL.hdr)[0] = dlo;
    reinterpret_cast<int4 *>(stage + SL.hdr)[1] = dhi;
    *reinterpret_cast<volatile int *>(stage + SL.seq) = index;
    mbar_arrive_expect_tx(full, (uint32_t)(uhi - ulo) + (uint32_t)(vhi - vlo) + extra_tx);
    bulk_g2s(smem_u32(stage + SL.units), reinterpret_cast<const unsigned char *>(t.units) + ulo,
             (uint32_t)(uhi - ulo), full);
    bulk_g2s(smem_u32(stage + SL.vals), reinterpret_cast<const unsigned char *>(t.values) + vlo,
             (uint32_t)(vhi - vlo), full);
}

// The consumer warps of k_stream: each takes the CTA's next block, waits for its stage, evaluates it
// and releases the stage; at the end it flushes its demand (and runs a pending price update).
template <int RT, bool PLAIN>
__device__ __forceinline__ void consume(const DevTable &t, const DevState &st, const DevPlan &pl, const SolveArgs &a,
                                        int round, int kind, unsigned char *smem, const StreamStageLayout &SL, int NS,
                                        uint32_t bars, int *grab, int nb, int lane)
{
    const int R = RT ? RT : t.R;
    auto full_bar = [&](int s) { return bars + 8u * (uint32_t)s; };
    auto empty_bar = [&](int s) { return bars + 8u * (uint32_t)(NS + s); };
    WarpCtx<RT, false> c;
    c.t = t;
    c.st = st;
    c.scen_warps = pl.scen_warps;
    c.a = a;
    c.round = round;
    c.R = R;
    c.rg = t.r_global;
    c.kind = PLAIN ? (int)PASS_ROUND : kind;
    c.want_min = PLAIN ? false : ((kind == PASS_FINAL) || (st.dual_trace != nullptr));
    c.want_hash = PLAIN ? false : ((kind == PASS_ROUND) && (st.hash_trace != nullptr));
    c.uniform_k = pl.uniform_k;
    c.log2_k = pl.uniform_k > 0 ? __ffs(pl.uniform_k) - 1 : 0;
    c.s = -1;
#pragma unroll
    for (int r = 0; r < Cols<RT>::N; ++r)
        c.acc[r] = 0;
    c.hacc = 0;
    c.defer = true;
    c.pend_s = -1;
    c.count_tiles = true;
    c.ntiles = 0;

    // prices, flags and demand accumulators were written by the previous kernel on the stream
    asm volatile("griddepcontrol.wait;" ::: "memory");
    bool failed = false;
    for (;;) {
        int i = 0;
        if (lane == 0)
            i = atomicAdd(grab, 1);   // the CTA's next block not yet taken
        i = __shfl_sync(FULL, i, 0);
        if (i >= nb)
            break;
        const int s = i % NS;
        const unsigned char *stage = smem + s * SL.bytes;
        // the stage's sequence word shows block i once its producer has issued it, which it does only
        // after the stage's previous block (i - NS) was consumed: the full barrier's current phase is
        // then block i's own, so the parity wait below cannot be satisfied by an older phase
        bool ok = true;
        if (lane == 0)
            ok = wait_word(reinterpret_cast<const volatile int *>(stage + SL.seq), i, st.err, a.wait_ms);
        if (!__shfl_sync(FULL, ok, 0) ||
            !__all_sync(FULL, wait_stage(full_bar(s), (uint32_t)((i / NS) & 1), st.err, a.wait_ms))) {
            failed = true;   // uniform decision; the CTA drains the copies in flight at its end
            break;
        }
        const TileDesc d = *reinterpret_cast<const TileDesc *>(stage + SL.hdr);
        if (d.scenario != c.s)
            enter_scenario<RT, false>(c, d.scenario, nullptr, lane);
        ++c.ntiles;
        if (!c.sp.skip) {
            const long long ulo = (d.opt_begin * R * 4) & ~15LL, vlo = (d.opt_begin * 8) & ~15LL;
            StagePtrs p;
            p.units = reinterpret_cast<const int32_t *>(stage + SL.units + (d.opt_begin * R * 4 - ulo));
            p.vals = reinterpret_cast<const double *>(stage + SL.vals + (d.opt_begin * 8 - vlo));
            p.grp = nullptr;
            p.off = nullptr;
            const int K = tile_run_k(d.flags);
            if (K > 128)
                process_tile_run4<RT, false, 2>(c, d, p, lane, K);
            else if (K >= 4)
                process_tile_run4<RT, false, 1>(c, d, p, lane, K);
            else
                process_tile_uniform<RT, false>(c, d, p, lane, K, K >> 1);
        }
        __syncwarp();
        if (lane == 0)
            mbar_arrive(empty_bar(s));
        run_pending(c, lane);
    }
    if (!failed) {
        flush<RT, false>(c, lane);
        run_pending(c, lane);
    }
}

template <int RT, bool PLAIN>
__global__ void __launch_bounds__((kStreamConsumers + kStreamProducers) * 32, 1)
    k_stream(DevTable t, DevState st, DevPlan pl, SolveArgs a, int round, int kind)
{
    extern __shared__ __align__(128) unsigned char smem[];
    // the next pass (a programmatic dependent) may start as soon as CTAs of this one finish; it
    // waits for this grid's completion before it reads any state
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
    const int R = RT ? RT : t.R;
    const StreamStageLayout SL = stream_stage_layout(pl.tile_opt, R);
    const int NS = stream_stages(pl.tile_opt, R);
    unsigned char *tail = smem + NS * SL.bytes;
    const uint32_t bars = smem_u32(tail);
    int *grab = reinterpret_cast<int *>(tail + 16 * NS);
    auto full_bar = [&](int s) { return bars + 8u * (uint32_t)s; };
    auto empty_bar = [&](int s) { return bars + 8u * (uint32_t)(NS + s); };
    __shared__ int skip_all;
    __shared__ int stage_last[ESP_STREAM_MAX_STAGES];   // the last block issued into each stage
    if (threadIdx.x == 0) {
        for (int s = 0; s < NS; ++s) {
            mbar_init(full_bar(s), 1);
            mbar_init(empty_bar(s), 1);
            stage_last[s] = -1;
            *reinterpret_cast<int *>(smem + s * SL.bytes + SL.seq) = -1;
        }
        fence_barrier_init();
        *grab = 0;
        // a wait of an earlier pass of this solve gave up: this pass does nothing (a flag set too
        // recently to be seen here only means the pass runs, with its own bounded waits)
        skip_all = (*reinterpret_cast<volatile unsigned int *>(st.err) & DEV_ERR_TIMEOUT) != 0;
    }
    __syncthreads();
    const int b0 = pl.cta_begin[blockIdx.x];
    const int nb = pl.cta_begin[blockIdx.x + 1] - b0;
    if (nb <= 0 || skip_all)
        return;

    if (wid >= kStreamConsumers) {
        // producer warp p: reads only the table and the plan, so it runs ahead of the previous
        // kernel's end. It issues the blocks p + P j, in order, into the stages p + P k it alone
        // fills (NS is a multiple of P): before block i it waits for the consumption of the stage's
        // previous block i - NS, which it issued itself after the one before was consumed, so the
        // empty barrier is at most one phase behind and its parity wait is unambiguous. Lane l holds
        // the descriptor of block p + P (batch + l), loaded a batch of 32 ahead of its use; lane 0
        // issues.
        const int p = wid - kStreamConsumers;
        const int4 *bd = reinterpret_cast<const int4 *>(pl.tiles + b0);
        int4 nlo = make_int4(0, 0, 0, 0), nhi = nlo;
        if (p + kStreamProducers * lane < nb) {
            nlo = __ldg(bd + 2 * (p + kStreamProducers * lane));
            nhi = __ldg(bd + 2 * (p + kStreamProducers * lane) + 1);
        }
        bool ok = true;
        for (int batch = 0; ok && p + kStreamProducers * batch < nb; batch += 32) {
            const int4 clo = nlo, chi = nhi;
            const int nx = p + kStreamProducers * (batch + 32 + lane);
            if (nx < nb) {   // the next batch's descriptors
                nlo = __ldg(bd + 2 * nx);
                nhi = __ldg(bd + 2 * nx + 1);
            }
            for (int k = 0; k < 32; ++k) {
                const int i = p + kStreamProducers * (batch + k);
                if (i >= nb)
                    break;
                const int4 dlo = make_int4(__shfl_sync(FULL, clo.x, k), __shfl_sync(FULL, clo.y, k),
                                           __shfl_sync(FULL, clo.z, k), __shfl_sync(FULL, clo.w, k));
                const int4 dhi = make_int4(__shfl_sync(FULL, chi.x, k), __shfl_sync(FULL, chi.y, k),
                                           __shfl_sync(FULL, chi.z, k), __shfl_sync(FULL, chi.w, k));
                const int s = i % NS;
                bool go = true;
                if (lane == 0) {
                    go = i < NS || wait_stage(empty_bar(s), (uint32_t)((i / NS - 1) & 1), st.err, a.wait_ms);
                    if (go) {
                        const uint32_t extra =
                            (blockIdx.x == 0 && i == 0 && round == 0 && kind == PASS_ROUND) ? a.hold_tx : 0u;
                        stage_last[s] = i;
                        issue_block(t, dlo, dhi, i, smem + s * SL.bytes, SL, full_bar(s), extra);
                    }
                }
                if (!__shfl_sync(FULL, go, 0)) {
                    ok = false;
                    break;
                }
            }
        }
    } else {
        consume<RT, PLAIN>(t, st, pl, a, round, kind, smem, SL, NS, full_bar(0), grab, nb, lane);
    }
    // Every copy issued into a stage has landed once the stage's latest phase is complete: always so
    // here unless a consumer gave up, in which case this waits (bounded) for the copies still in
    // flight before the CTA may exit. The latest phase of a stage is never followed by another one,
    // so this wait cannot mistake an older phase for it.
    __syncthreads();
    if (threadIdx.x == 0)
        for (int s = 0; s < NS; ++s)
            if (stage_last[s] >= 0)
                wait_stage(full_bar(s), (uint32_t)((stage_last[s] / NS) & 1), st.err, a.wait_ms);
}

template <int RT>
struct StreamKernels {
    static const void *plain() { return reinterpret_cast<const void *>(&k_stream<RT, true>); }
    static const void *other() { return reinterpret_cast<const void *>(&k_stream<RT, false>); }
    static void launch(bool plain_pass, int grid, int smem, cudaStream_t stream, const DevTable &t,
                       const DevState &st, const DevPlan &pl, const SolveArgs &a, int round, int kind, bool pdl)
    {
        cudaLaunchConfig_t cfg = {};
        cfg.gridDim = dim3((unsigned)grid);
        cfg.blockDim = dim3((kStreamConsumers + kStreamProducers) * 32);
        cfg.dynamicSmemBytes = (size_t)smem;
        cfg.stream = stream;
        cudaLaunchAttribute attr[1];
        attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
        attr[0].val.programmaticStreamSerializationAllowed = 1;
        cfg.attrs = attr;
        cfg.numAttrs = pdl ? 1 : 0;
        if (plain_pass)
            cudaLaunchKernelEx(&cfg, k_stream<RT, true>, t, st, pl, a, round, kind);
        else
            cudaLaunchKernelEx(&cfg, k_stream<RT, false>, t, st, pl, a, round, kind);
    }
};

template <typename F>
auto dispatch_stream(int R, F &&f)
{
    switch (R) {
    case 4: return f(StreamKernels<4>());
    case 6: return f(StreamKernels<6>());
    case 8: return f(StreamKernels<8>());
    default: return f(StreamKernels<0>());
    }
}

}  // namespace

int stream_ctas_per_sm(int R)
{
    // at least two stages per producer warp
    if (stream_stages(stream_stage_opt(R), R) < 2 * kStreamProducers)
        return 0;
    const int smem = stream_smem_bytes(stream_stage_opt(R), R);
    return dispatch_stream(R, [&](auto k) -> int {
        using K = decltype(k);
        if (cudaFuncSetAttribute(K::plain(), cudaFuncAttributeMaxDynamicSharedMemorySize, smem) != cudaSuccess ||
            cudaFuncSetAttribute(K::other(), cudaFuncAttributeMaxDynamicSharedMemorySize, smem) != cudaSuccess) {
            cudaGetLastError();
            return 0;
        }
        const int threads = (kStreamConsumers + kStreamProducers) * 32;
        int n = 0, m = 0;
        if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, K::plain(), threads, smem) != cudaSuccess ||
            cudaOccupancyMaxActiveBlocksPerMultiprocessor(&m, K::other(), threads, smem) != cudaSuccess) {
            cudaGetLastError();
            return 0;
        }
        return n < m ? n : m;
    });
}

cudaError_t launch_stream(const DevTable &t, const DevState &st, const DevPlan &pl, const SolveArgs &a, int round,
                          PassKind kind, int grid, cudaStream_t stream, bool pdl)
{
    const int smem = stream_smem_bytes(pl.tile_opt, t.R);
    const bool plain = kind == PASS_ROUND && st.hash_trace == nullptr && st.dual_trace == nullptr;
    dispatch_stream(t.R, [&](auto k) -> int {
        decltype(k)::launch(plain, grid, smem, stream, t, st, pl, a, round, kind, pdl);
        return 0;
    });
    return cudaGetLastError();
}

}  // namespace esp
