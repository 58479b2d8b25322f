// Device kernels of the ESP tatonnement (Sec. 3.2 of the paper) for sm_103a.
//
// One evaluation pass (a best response of every job, Sec. 3.2.2; Eq. esp_score without Gamma) runs
// as warps that each own a static list of tiles. A tile is a run of whole jobs of one scenario (or
// one chunk of a job larger than a tile); its option bytes are contiguous in HBM and arrive in the
// warp's shared-memory stage by 1-D bulk copies (cp.async.bulk + mbarrier), one tile ahead of the
// tile being evaluated.
//
// Exactness. The returned choice is the lexicographic minimum of (s, local index) with
//   s = fma(p_{R-1}, u_{R-1}, ... fma(p_0, u_0, -v))         (fp64, r = 0 .. R-1)
// exactly as the oracle computes it. GB300 runs fp64 at a small fraction of its fp32 rate, so each
// option is first scored in fp32, q = the same chain in fp32, with |q - s| <= E for every option of
// the scenario (E from the bound below). A job whose smallest q beats every other q by more than 2E
// has that option as its exact argmin; otherwise every option with q <= m1 + 2E (rounded up) is
// rescored in fp64 and the exact lexicographic minimum is taken. Proof: s_i <= s_w implies
// q_i - E <= s_i <= s_w <= q_w + E = m1 + E. The bound (fp32 unit roundoff u = 2^-24, all
// magnitudes M = |v| + sum_r p_r u_r, prices rounded to fp32 once, v truncated to fp32 (error
// below 2u|v|, or below 2^-100 when |v| < 2^-100), units exact, R fused steps, fp64 error
// R 2^-53 M, subnormal absolute error below 2^-100 in total) is
//   |q - s| <= (R + 4) u M (1 + small) + 2^-99 ;   E = (4R + 16) u M_s + 2^-99,
// with M_s = max|v| + sum_r max p_r * max u_r over the scenario, a factor of about 4 to spare.
// A scenario whose prices or values leave [2^-100, 2^100] in magnitude is evaluated in fp64 only.
//
// Aggregation. Demands of the chosen options are summed in int64 registers per lane, reduced
// across the warp and added with one 64-bit atomic per priced resource per warp and scenario:
// integer addition is associative, so U is identical on every run.

#include <algorithm>
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



__global__ void k_init(DevTable t, DevState st, SolveArgs a, const double *lambda0)
{
    const int lane = threadIdx.x & 31;
    const int s = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
    if (s >= t.S)
        return;
    const int P = t.P;
    for (int k = lane; k < P; k += 32) {
        const double l0 = lambda0 ? lambda0[(size_t)s * P + k] : 0.0;
        st.lam[(size_t)s * P + k] = l0;
        st.U[(size_t)s * P + k] = 0ull;
        st.U_final[(size_t)s * P + k] = 0ull;
        if (st.lam_trace)
            st.lam_trace[((size_t)s * (a.T + 1)) * P + k] = l0;
    }
    if (lane == 0) {
        st.hash[s] = 0ull;
        st.arrive[s] = 0u;
        st.rounds_run[s] = 0;
        st.converged[s] = 0;
        st.status[s] = 0;
        st.frozen[s] = 0;
        st.best_dual[s] = INFINITY;
    }
    __syncwarp();
    set_prices<8>(t, st, a, s, lane);
}

// Separate price-update launch (used when no warp owns tiles, e.g. J = 0).
__global__ void k_update(DevTable t, DevState st, SolveArgs a, int round)
{
    const int lane = threadIdx.x & 31;
    const int s = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
    if (s >= t.S || st.frozen[s])
        return;
    update_scenario<8>(t, st, a, s, round, lane);
}

// Data of tile-local option o (stage) or of job option o (global, gfirst = the job's first option).

// Asks L2 for the option bytes of tile d (lane 0 only), a few tiles before the stage copy of the
// same bytes is issued: the DRAM latency is then hidden by L2 rather than by shared memory.
__device__ __forceinline__ void prefetch_tile(const DevTable &t, const TileDesc &d)
{
    const int R = t.R;
    const int64_t ub = d.opt_begin * R * 4, ue = (d.opt_begin + d.n_opt) * R * 4;
    const int64_t ulo = ub & ~int64_t(15), uhi = (ue + 15) & ~int64_t(15);
    const int64_t vb = d.opt_begin * 8, ve = (d.opt_begin + d.n_opt) * 8;
    const int64_t vlo = vb & ~int64_t(15), vhi = (ve + 15) & ~int64_t(15);
    prefetch_l2(reinterpret_cast<const unsigned char *>(t.units) + ulo, (uint32_t)(uhi - ulo));
    prefetch_l2(reinterpret_cast<const unsigned char *>(t.values) + vlo, (uint32_t)(vhi - vlo));
}

// Chunk tile of a job larger than a tile: all its options belong to one job, so no segmentation is


// Issues the bulk copies of tile d into a stage; lane 0 only (issuing the copies from several lanes
// at once measured slower). Uniform tables and runs of the sorted layout need no job offsets.
__device__ __forceinline__ void issue_tile(const DevTable &t, const TileDesc &d, unsigned char *stage,
                                           const StageLayout &SL, uint32_t bar, bool need_offsets, uint32_t extra_tx = 0)
{
    const int R = t.R;
    if (t.il) {   // the tile's units and values are adjacent: one copy (its start is 16-byte aligned)
        const int64_t W = 4 * R + 8;
        const int64_t b = d.opt_begin * W, e = ((d.opt_begin + d.n_opt) * W + 15) & ~int64_t(15);
        fence_proxy_async();
        mbar_arrive_expect_tx(bar, (uint32_t)(e - b) + extra_tx);
        bulk_g2s(smem_u32(stage + SL.units), t.il + b, (uint32_t)(e - b), bar);
        return;
    }
    const int64_t ub = d.opt_begin * R * 4, ue = (d.opt_begin + d.n_opt) * R * 4;
    const int64_t ulo = ub & ~int64_t(15), uhi = (ue + 15) & ~int64_t(15);
    const int64_t vb = d.opt_begin * 8, ve = (d.opt_begin + d.n_opt) * 8;
    const int64_t vlo = vb & ~int64_t(15), vhi = (ve + 15) & ~int64_t(15);
    uint32_t total = (uint32_t)(uhi - ulo) + (uint32_t)(vhi - vlo);
    int64_t olo = 0, ohi = 0, glo = 0, ghi = 0;
    const bool offs = need_offsets && !(d.flags & (TILE_BIG | TILE_RUN));
    if (offs) {
        const int64_t ob = d.job_begin * 8, oe = (d.job_begin + d.n_job + 1) * 8;
        olo = ob & ~int64_t(15);
        ohi = (oe + 15) & ~int64_t(15);
        total += (uint32_t)(ohi - olo);
    }
    if (t.group) {
        const int64_t gb = d.opt_begin * 2, ge = (d.opt_begin + d.n_opt) * 2;
        glo = gb & ~int64_t(15);
        ghi = (ge + 15) & ~int64_t(15);
        total += (uint32_t)(ghi - glo);
    }
    fence_proxy_async();
    mbar_arrive_expect_tx(bar, total + extra_tx);
    const unsigned char *ubase = reinterpret_cast<const unsigned char *>(t.units);
    const unsigned char *vbase = reinterpret_cast<const unsigned char *>(t.values);
    bulk_g2s(smem_u32(stage + SL.units), ubase + ulo, (uint32_t)(uhi - ulo), bar);
    bulk_g2s(smem_u32(stage + SL.vals), vbase + vlo, (uint32_t)(vhi - vlo), bar);
    if (offs)
        bulk_g2s(smem_u32(stage + SL.off), reinterpret_cast<const unsigned char *>(t.job_off) + olo,
                 (uint32_t)(ohi - olo), bar);
    if (t.group)
        bulk_g2s(smem_u32(stage + SL.grp), reinterpret_cast<const unsigned char *>(t.group) + glo,
                 (uint32_t)(ghi - glo), bar);
}

// CTAs per SM the evaluation kernel's register budget must allow.
// CTAs per SM the evaluation kernel's register budget must allow: the uniform and runs-only
// instantiations (no segmented-scan path) as many as the general one's shared memory would.
template <int RT, int MODE>
constexpr int pass_min_ctas()
{
    return MODE == kModeUniform ? ((RT == 4 || RT == 6) ? kMinCtasPerSmNarrow : kMinCtasPerSm)
           : MODE == kModeRuns  ? kMinCtasPerSmRuns
                                : kMinCtasPerSmGeneral;
}

template <int RT, bool G, int MODE, bool PLAIN>
__global__ void __launch_bounds__(kWarpsPerCta * 32, pass_min_ctas<RT, MODE>()) k_pass(DevTable t, DevState st, DevPlan pl,
                                                                          SolveArgs a, int round, int kind)
{
    extern __shared__ __align__(128) unsigned char smem[];
    // a pass launched as a programmatic dependent of this one may start its CTAs as soon as slots
    // free up; it waits (griddepcontrol.wait below) for this grid's completion before reading state
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
    const int w = blockIdx.x * kWarpsPerCta + wid;
    if (w >= pl.n_warps)
        return;
    const int k_begin = pl.warp_begin[w], k_end = pl.warp_begin[w + 1];
    if (k_begin >= k_end)
        return;
    // a wait of an earlier pass of this solve gave up: this warp does nothing (a flag set too recently
    // to be seen here only means the warp runs, with its own bounded waits)
    if (__any_sync(FULL, (*reinterpret_cast<volatile unsigned int *>(st.err) & DEV_ERR_TIMEOUT) != 0))
        return;

    constexpr bool UNI = MODE == kModeUniform;
    const WarpSmem WS = warp_smem(pl.tile_opt, t.R, G, t.P, MODE == kModeGeneral);
    const StageLayout SL = stage_layout(pl.tile_opt, t.R, G, MODE == kModeGeneral);
    unsigned char *wsm = smem + (size_t)wid * WS.bytes;
    float *p32s = reinterpret_cast<float *>(wsm + WS.p32);
    const uint32_t bar0 = smem_u32(wsm + WS.bars);
    const bool need_offsets = MODE == kModeGeneral;

    WarpCtx<RT, G> c;
    c.t = t;
    c.st = st;
    c.scen_warps = pl.scen_warps;
    c.a = a;
    c.round = round;
    c.R = RT ? RT : t.R;
    c.rg = t.r_global;
    // PLAIN: a round pass without traces (the hot case), with every per-pass choice a constant
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

    if (lane == 0) {
        for (int s = 0; s < kStages; ++s)
            mbar_init(bar0 + 8 * s, 1);
        fence_barrier_init();
    }
    __syncwarp();

    // Tile descriptors reach the warp's ring in blocks of kDescBlock: one cp.async of 16 bytes per
    // lane fetches a block, issued a whole block before its first tile is issued, so no global
    // load sits on the per-tile path. Block b uses ring slots (b & 1) * kDescBlock onwards.
    TileDesc *ring = reinterpret_cast<TileDesc *>(wsm + WS.descs);
    const unsigned char *tiles_b = reinterpret_cast<const unsigned char *>(pl.tiles);
    auto fetch_block = [&](int first) {
        const int ti = first + (lane >> 1);
        if (lane < 2 * kDescBlock && ti < k_end) {
            const uint32_t dst = smem_u32(ring + ((ti - k_begin) & (kDescRing - 1))) + 16u * (lane & 1);
            asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(dst),
                         "l"(tiles_b + (size_t)ti * sizeof(TileDesc) + 16 * (lane & 1))
                         : "memory");
        }
        asm volatile("cp.async.commit_group;" ::: "memory");
    };
    auto wait_blocks = [&]() {
        asm volatile("cp.async.wait_group 0;" ::: "memory");
        __syncwarp();
    };
    fetch_block(k_begin);
    fetch_block(k_begin + kDescBlock);
    wait_blocks();

    // prologue: the first kStages-1 tiles in flight (lane 0 issues every copy)
    int issued = k_begin;
    while (issued < k_end && issued < k_begin + kStages - 1) {
        const int sidx = (issued - k_begin) % kStages;
        if (lane == 0)
            issue_tile(t, ring[(issued - k_begin) & (kDescRing - 1)], wsm + sidx * SL.bytes, SL, bar0 + 8 * sidx,
                       need_offsets, (w == 0 && issued == k_begin && round == 0 && kind == PASS_ROUND) ? a.hold_tx : 0u);
        ++issued;
    }
    __syncwarp();
    if (lane == 0)
        for (int k = issued; k < k_end && k < k_begin + kPrefetchTiles; ++k)
            prefetch_tile(t, pl.tiles[k]);
    // everything above reads only the table and the plan; prices, flags and the demand accumulators
    // were written by the previous kernel on the stream, which is complete after this wait (a no-op
    // for an ordinary launch)
    asm volatile("griddepcontrol.wait;" ::: "memory");
    int64_t big_first = 0;
    Best big_carry = best_none();
    Best big_priv = best_none();     // lane-private state of a chunked job
    int failed_at = -1;
    for (int k = k_begin; k < k_end; ++k) {
        if (issued < k_end) {   // refill the stage the previous tile used
            if (((issued - k_begin) & (kDescBlock - 1)) == 0)
                wait_blocks();  // the block that starts with tile `issued` has landed
            if (lane == 0) {
                const int sidx = (issued - k_begin) % kStages;
                issue_tile(t, ring[(issued - k_begin) & (kDescRing - 1)], wsm + sidx * SL.bytes, SL,
                           bar0 + 8 * sidx, need_offsets);
                if (kPrefetchTiles > 0 && k + kPrefetchTiles < k_end)
                    prefetch_tile(t, pl.tiles[k + kPrefetchTiles]);
            }
            ++issued;
        }
        const TileDesc d = ring[(k - k_begin) & (kDescRing - 1)];
        const int sidx = (k - k_begin) % kStages;
        const uint32_t parity = (uint32_t)(((k - k_begin) / kStages) & 1);
        if (!__all_sync(FULL, wait_stage(bar0 + 8 * sidx, parity, st.err, a.wait_ms))) {   // uniform decision
            failed_at = k;
            break;
        }
        if (d.scenario != c.s)
            enter_scenario<RT, G>(c, d.scenario, p32s, lane);
        if (!c.sp.skip) {
            const StagePtrs ptrs = t.il ? stage_ptrs_il(d, wsm + sidx * SL.bytes, SL, c.R)
                                        : stage_ptrs(d, wsm + sidx * SL.bytes, SL, c.R);
            if (UNI && c.uniform_k >= 4)
                process_tile_uniform4<RT, G>(c, d, ptrs, lane);
            else if (UNI)
                process_tile_uniform<RT, G>(c, d, ptrs, lane, c.uniform_k, c.log2_k);
            else if (d.flags & TILE_BIG)
                process_tile_bigchunk<RT, G>(c, d, ptrs, big_first, big_priv, lane);
            else if (!G && (d.flags & TILE_RUN) && tile_run_k(d.flags) >= 4)
                process_tile_run4<RT, G>(c, d, ptrs, lane, tile_run_k(d.flags));
            else if (!G && (d.flags & TILE_RUN))
                process_tile_uniform<RT, G>(c, d, ptrs, lane, tile_run_k(d.flags), tile_run_k(d.flags) >> 1);
            else if (MODE == kModeGeneral)
                process_tile_general<RT, G>(c, d, ptrs, big_first, big_carry, lane);
        }
        __syncwarp();
        // the last tile of a block is done (issued and evaluated): its slots take the block after next
        if (((k - k_begin) & (kDescBlock - 1)) == kDescBlock - 1)
            fetch_block(k + 1 + kDescBlock);
    }
    asm volatile("cp.async.wait_group 0;" ::: "memory");
    if (failed_at < 0) {
        flush<RT, G>(c, lane);
    } else {
        // a copy never completed: wait (bounded) for every copy still in flight, then leave
        for (int k = failed_at; k < issued; ++k) {
            const int sidx = (k - k_begin) % kStages;
            wait_stage(bar0 + 8 * sidx, (uint32_t)(((k - k_begin) / kStages) & 1), st.err, a.wait_ms);
        }
    }
}

__global__ void k_objectives(DevTable t, DevState st, SolveArgs a)
{
    const int lane = threadIdx.x & 31;
    const int s = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
    if (s >= t.S)
        return;
    const int P = t.P, J = t.J;
    const size_t sp = (size_t)s * P;
    double pv = 0.0, pm = 0.0, lc = 0.0;
    for (int j = lane; j < J; j += 32) {
        pv += st.job_val[(size_t)s * J + j];
        pm += -st.job_min[(size_t)s * J + j];
    }
    bool feas = true;
    for (int k = lane; k < P; k += 32) {
        lc += (a.mode == 1) ? st.lam[sp + k] : st.lam[sp + k] * (double)t.cap[sp + k];
        feas &= (long long)st.U_final[sp + k] <= t.cap[sp + k];
    }
    const double primal = warp_sum_fixed(pv);
    const double g = warp_sum_fixed(pm) + warp_sum_fixed(lc);
    feas = __all_sync(FULL, feas);
    if (lane == 0) {
        st.primal[s] = primal;
        st.dual[s] = g;
        st.feasible[s] = feas ? 1 : 0;
        const double bd = st.best_dual[s];
        st.best_dual[s] = (st.dual_trace && bd < g) ? bd : g;
        if (st.dual_trace)
            st.dual_trace[(size_t)s * (a.T + 1) + st.rounds_run[s]] = g;
        if (st.lam_trace) {
            // the final prices also close the trace at row rounds_run (already written by the update)
        }
    }
}
// Both instantiations (plain round pass and the general one) of a table shape.
template <int RT, bool G, int MODE>
struct PassKernels {
    static const void *plain() { return reinterpret_cast<const void *>(&k_pass<RT, G, MODE, true>); }
    static const void *other() { return reinterpret_cast<const void *>(&k_pass<RT, G, MODE, false>); }
    // pdl: programmatic dependent launch, so the pass's CTAs may start (and stage their first tiles)
    // while the previous kernel on the stream finishes; the kernel waits for it before reading state
    static void launch(bool plain, int grid, int smem, cudaStream_t stream, const DevTable &t, const DevState &st,
                       const DevPlan &pl, const SolveArgs &a, int round, int kind, bool pdl)
    {
        cudaLaunchConfig_t cfg = {};
        cfg.gridDim = dim3((unsigned)grid);
        cfg.blockDim = dim3(kWarpsPerCta * 32);
        cfg.dynamicSmemBytes = (size_t)smem;
        cfg.stream = stream;
        cudaLaunchAttribute attr[1];
        attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
        attr[0].val.programmaticStreamSerializationAllowed = 1;
        cfg.attrs = attr;
        cfg.numAttrs = pdl ? 1 : 0;
        if (plain)
            cudaLaunchKernelEx(&cfg, k_pass<RT, G, MODE, true>, t, st, pl, a, round, kind);
        else
            cudaLaunchKernelEx(&cfg, k_pass<RT, G, MODE, false>, t, st, pl, a, round, kind);
    }
};

// Calls f(PassKernels<RT, G, MODE>()) for the instantiation that serves this table shape (grouped
// tables are always general).
template <typename F>
auto dispatch_shape(int R, bool grouped, int mode, F &&f)
{
    if (grouped) {
        switch (R) {
        case 4: return f(PassKernels<4, true, kModeGeneral>());
        case 6: return f(PassKernels<6, true, kModeGeneral>());
        case 8: return f(PassKernels<8, true, kModeGeneral>());
        default: return f(PassKernels<0, true, kModeGeneral>());
        }
    }
    if (mode == kModeUniform) {
        switch (R) {
        case 4: return f(PassKernels<4, false, kModeUniform>());
        case 6: return f(PassKernels<6, false, kModeUniform>());
        case 8: return f(PassKernels<8, false, kModeUniform>());
        default: return f(PassKernels<0, false, kModeUniform>());
        }
    }
    if (mode == kModeRuns) {
        switch (R) {
        case 4: return f(PassKernels<4, false, kModeRuns>());
        case 6: return f(PassKernels<6, false, kModeRuns>());
        case 8: return f(PassKernels<8, false, kModeRuns>());
        default: return f(PassKernels<0, false, kModeRuns>());
        }
    }
    switch (R) {
    case 4: return f(PassKernels<4, false, kModeGeneral>());
    case 6: return f(PassKernels<6, false, kModeGeneral>());
    case 8: return f(PassKernels<8, false, kModeGeneral>());
    default: return f(PassKernels<0, false, kModeGeneral>());
    }
}

}  // namespace

int pass_smem_bytes(int R, bool grouped, int mode, int P, int tile_opt)
{
    return kWarpsPerCta * warp_smem(tile_opt, R, grouped, P, grouped || mode == kModeGeneral).bytes;
}

int pass_ctas_per_sm(int R, bool grouped, int mode, int P, int tile_opt)
{
    const int smem = pass_smem_bytes(R, grouped, mode, P, tile_opt);
    return dispatch_shape(R, grouped, mode, [&](auto k) -> int {
        using K = decltype(k);
        if (cudaFuncSetAttribute(K::plain(), cudaFuncAttributeMaxDynamicSharedMemorySize, smem) != cudaSuccess ||
            cudaFuncSetAttribute(K::other(), cudaFuncAttributeMaxDynamicSharedMemorySize, smem) != cudaSuccess)
            return 0;
        int n = 0;
        if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, K::plain(), kWarpsPerCta * 32, smem) != cudaSuccess)
            return 0;
        int m = 0;
        if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&m, K::other(), kWarpsPerCta * 32, smem) != cudaSuccess)
            return 0;
        return n < m ? n : m;
    });
}

cudaError_t launch_init(const DevTable &t, const DevState &st, const SolveArgs &a, const double *lambda0,
                        cudaStream_t stream)
{
    const int wpb = 4;
    k_init<<<(t.S + wpb - 1) / wpb, 32 * wpb, 0, stream>>>(t, st, a, lambda0);
    return cudaGetLastError();
}

cudaError_t launch_pass(const DevTable &t, const DevState &st, const DevPlan &pl, const SolveArgs &a, int round,
                        PassKind kind, int grid, cudaStream_t stream, bool pdl)
{
    const bool grouped = t.group != nullptr;
    const int mode = pass_mode(pl);
    const int smem = pass_smem_bytes(t.R, grouped, mode, t.P, pl.tile_opt);
    const bool plain = kind == PASS_ROUND && st.hash_trace == nullptr && st.dual_trace == nullptr;
    dispatch_shape(t.R, grouped, mode, [&](auto k) -> int {
        decltype(k)::launch(plain, grid, smem, stream, t, st, pl, a, round, kind, pdl);
        return 0;
    });
    return cudaGetLastError();
}

cudaError_t launch_update(const DevTable &t, const DevState &st, const SolveArgs &a, int round, cudaStream_t stream)
{
    const int wpb = 4;
    k_update<<<(t.S + wpb - 1) / wpb, 32 * wpb, 0, stream>>>(t, st, a, round);
    return cudaGetLastError();
}

cudaError_t launch_objectives(const DevTable &t, const DevState &st, const SolveArgs &a, cudaStream_t stream)
{
    const int wpb = 4;
    k_objectives<<<(t.S + wpb - 1) / wpb, 32 * wpb, 0, stream>>>(t, st, a);
    return cudaGetLastError();
}

}  // namespace esp
