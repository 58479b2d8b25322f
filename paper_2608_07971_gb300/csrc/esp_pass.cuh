// The per-warp evaluation-pass kernel of the ESP tatonnement (Sec. 3.2.2; Eq. esp_score without
// Gamma) for sm_103a, shared by the two translation units that instantiate it: esp_kernels.cu (units
// staged as integers) and esp_kernels_f32.cu (units staged as fp32, for tables whose units are all
// below 2^23). The exactness argument and the aggregation are stated in esp_kernels.cu.
#pragma once

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

// F: the stage holds units as fp32 bit patterns (DevTable::il_f32), read by the screen as they are.
template <int RT, bool G, int MODE, bool PLAIN, bool F>
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
    c.persist = false;
    c.scen_tiles = nullptr;
    c.ntiles = 0;
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
                process_tile_uniform4<RT, G, F>(c, d, ptrs, lane);
            else if (UNI)
                process_tile_uniform<RT, G, F>(c, d, ptrs, lane, c.uniform_k, c.log2_k);
            else if (d.flags & TILE_BIG)
                process_tile_bigchunk<RT, G, F>(c, d, ptrs, big_first, big_priv, lane);
            else if (!G && (d.flags & TILE_RUN) && tile_run_k(d.flags) >= 4)
                process_tile_run4<RT, G, F>(c, d, ptrs, lane, tile_run_k(d.flags));
            else if (!G && (d.flags & TILE_RUN))
                process_tile_uniform<RT, G, F>(c, d, ptrs, lane, tile_run_k(d.flags), tile_run_k(d.flags) >> 1);
            else if (MODE == kModeGeneral)
                process_tile_general<RT, G, F>(c, d, ptrs, big_first, big_carry, lane);
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

// Both instantiations (plain round pass and the general one) of a table shape.
template <int RT, bool G, int MODE, bool F = false>
struct PassKernels {
    static const void *plain() { return reinterpret_cast<const void *>(&k_pass<RT, G, MODE, true, F>); }
    static const void *other() { return reinterpret_cast<const void *>(&k_pass<RT, G, MODE, false, F>); }
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
            cudaLaunchKernelEx(&cfg, k_pass<RT, G, MODE, true, F>, t, st, pl, a, round, kind);
        else
            cudaLaunchKernelEx(&cfg, k_pass<RT, G, MODE, false, F>, t, st, pl, a, round, kind);
    }
};

// ---------------------------------------------------------------------------------------------
// Persistent pass: rounds 0 .. T-1 of a solve in one cooperative launch.
//
// Between two round passes a kernel boundary costs the whole GPU the slowest warp's tail, the next
// pass's ramp-up and the launch gap (measured at about 21 us per round on the what-if batch and
// 39 us on the heavy-tailed table, against 160 and 300 us of streaming). Here the only dependence
// left is the true one: scenario s may be evaluated in round r once its r-th price update is done.
// The last warp to finish s in a round applies Eq. price_update (as in the round pass) and then
// releases ver[s] = r + 1; a warp entering s in round r acquire-polls ver[s] >= r.
// Work items are (round, plan range) pairs, q = round * n_ranges + k, taken from one counter in
// increasing order by whichever warp is free (static assignments measured 10% slower: some warps run
// systematically slower than others); the k-th range handed out in a round is item_order[k], the
// ranges sorted by the scenario of their first tile (a sorted layout keeps a scenario's tiles in
// three parts of the table). The items of a scenario's next round are therefore handed out about a
// round after its current ones: a warp waits only when another is most of a round late with one. A warp takes items ahead of the
// one it evaluates, so that its copy pipeline runs on without a gap across items (the table does
// not depend on prices).
// Deadlock-free: every CTA is co-resident (cooperative launch); an item depends only on items of
// smaller index, and the smallest item not yet done is some warp's current item, whose
// dependencies are all done. Every wait is bounded.

// Bounded wait of a warp until scenario s has had `round` price updates (ver[s] >= round). Every lane
// polls the word with relaxed loads (one transaction per poll) and, once all see it, reads it once
// more with acquire semantics, so that each lane's later reads of the scenario's prices and bound are
// ordered after the update that released them. The poll spins (each load is an L2 round trip) and
// sleeps only after a long spin: a sleep can last far longer than asked, and a woken waiter would
// then lag its scenario by that much. Gives up when another wait flagged a timeout, or after
// limit_ms of the global timer (flagging one). The result is warp-uniform.
__device__ __forceinline__ bool wait_version(const unsigned int *ver, int s, int round, unsigned int *err,
                                             uint32_t limit_ms, unsigned long long *stats)
{
    auto seen = [&](bool acquire) {
        unsigned int v;
        if (acquire)
            asm volatile("ld.acquire.gpu.u32 %0, [%1];" : "=r"(v) : "l"(ver + s) : "memory");
        else
            asm volatile("ld.relaxed.gpu.u32 %0, [%1];" : "=r"(v) : "l"(ver + s) : "memory");
        return __all_sync(FULL, v >= (unsigned int)round);
    };
    if (seen(true))
        return true;
    const uint64_t t0 = __shfl_sync(FULL, global_ns(), 0);
    const uint64_t limit = (uint64_t)limit_ms * 1000000ull;
    bool ok = false;
    for (uint32_t it = 1;; ++it) {
        if (seen(false)) {
            ok = seen(true);   // the value only grows: the acquire read sees it too
            if (ok)
                break;
        }
        if ((it & 63) == 0) {
            unsigned int e;
            asm volatile("ld.relaxed.gpu.u32 %0, [%1];" : "=r"(e) : "l"(err) : "memory");
            if (__any_sync(FULL, (e & DEV_ERR_TIMEOUT) != 0))
                break;
            if (__shfl_sync(FULL, (global_ns() - t0 > limit) ? 1 : 0, 0)) {
                if ((threadIdx.x & 31) == 0)
                    atomicOr(err, DEV_ERR_TIMEOUT);
                break;
            }
            if (it >= 4096)
                __nanosleep(256);
        }
    }
    if ((threadIdx.x & 31) == 0) {   // the time this wait polled (esp_debug_persist_waits)
        atomicAdd(stats + 2, (unsigned long long)(global_ns() - t0));
        atomicAdd(stats + 3, 1ull);
    }
    return ok;
}

template <int RT, int MODE, bool F>
__global__ void __launch_bounds__(kWarpsPerCta * 32, pass_min_ctas<RT, MODE>())
    k_pass_persist(DevTable t, DevState st, DevPlan pl, SolveArgs a, int n_rounds)
{
    constexpr bool G = false;
    constexpr bool UNI = MODE == kModeUniform;
    extern __shared__ __align__(128) unsigned char smem[];
    const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
    const bool first_warp = blockIdx.x == 0 && wid == 0;
    const WarpSmem WS = warp_smem(pl.tile_opt, t.R, false, t.P, false);
    const StageLayout SL = stage_layout(pl.tile_opt, t.R, false, false);
    unsigned char *wsm = smem + (size_t)wid * (WS.bytes + kPersistQueueBytes);
    // the warp's queue of taken items: item index, first tile, tiles, first virtual tile
    int *q_item = reinterpret_cast<int *>(wsm + WS.bytes);
    int *q_beg = q_item + kPersistQueue, *q_len = q_beg + kPersistQueue, *q_vs = q_len + kPersistQueue;
    const uint32_t bar0 = smem_u32(wsm + WS.bars);
    const int NR = pl.n_warps;
    const int64_t Q = (int64_t)n_rounds * NR;   // items (the host keeps Q below 2^31)
    if (__any_sync(FULL, (*reinterpret_cast<volatile unsigned int *>(st.err) & DEV_ERR_TIMEOUT) != 0))
        return;

    // queue state (warp-uniform): items [qh, qt) taken, their tiles are virtual tiles [.., known).
    // Lane 0 asks the counter for the item after the next one as soon as it takes the next one, so
    // that the atomic's latency is hidden by the current item's tiles.
    int qh = 0, qt = 0, known = 0;
    bool exhausted = false;
    unsigned int pend = 0;
    if (lane == 0)
        pend = atomicAdd(st.work, 1u);
    // takes items until the virtual tiles up to `need` are known (or none is left)
    auto take_until = [&](int need) {
        while (known < need && !exhausted && qt - qh < kPersistQueue) {
            int q = 0, b = 0, n = 0;
            if (lane == 0) {
                q = (int)pend;
                if ((int64_t)q < Q)
                    pend = atomicAdd(st.work, 1u);
                if ((int64_t)q < Q) {
                    const int i = __ldg(pl.item_order + q % NR);
                    b = __ldg(pl.warp_begin + i);
                    n = __ldg(pl.warp_begin + i + 1) - b;
                }
            }
            q = __shfl_sync(FULL, q, 0);
            b = __shfl_sync(FULL, b, 0);
            n = __shfl_sync(FULL, n, 0);
            if ((int64_t)q >= Q) {
                exhausted = true;
            } else if (n > 0) {
                const int slot = qt % kPersistQueue;
                if (lane == 0) {
                    q_item[slot] = q;
                    q_beg[slot] = b;
                    q_len[slot] = n;
                    q_vs[slot] = known;
                }
                ++qt;
                known += n;
            }
        }
        __syncwarp();
    };
    // tile of virtual tile vv (known)
    auto tile_at = [&](int vv) -> int {
        int k = qh;
        while (vv >= q_vs[k % kPersistQueue] + q_len[k % kPersistQueue])
            ++k;
        const int slot = k % kPersistQueue;
        return q_beg[slot] + (vv - q_vs[slot]);
    };
    // the descriptor of virtual tile vv into its ring slot (two lanes, one cp.async group)
    TileDesc *ring = reinterpret_cast<TileDesc *>(wsm + WS.descs);
    const unsigned char *tiles_b = reinterpret_cast<const unsigned char *>(pl.tiles);
    auto fetch_desc = [&](int vv) {
        if (lane < 2 && vv < known) {
            const int ti = tile_at(vv);
            const uint32_t dst = smem_u32(ring + (vv & (kDescRing - 1))) + 16u * lane;
            asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(dst),
                         "l"(tiles_b + (size_t)ti * sizeof(TileDesc) + 16 * lane)
                         : "memory");
        }
        asm volatile("cp.async.commit_group;" ::: "memory");
    };

    WarpCtx<RT, G> c;
    c.persist = true;
    c.scen_tiles = pl.scen_tiles;
    c.ntiles = 0;
    c.t = t;
    c.st = st;
    c.scen_warps = pl.scen_warps;
    c.a = a;
    c.round = 0;
    c.R = RT ? RT : t.R;
    c.rg = t.r_global;
    c.kind = (int)PASS_ROUND;
    c.want_min = false;
    c.want_hash = false;
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

    take_until(kStages + 1);
    if (known == 0)
        return;
    // prologue: descriptors of the first kStages tiles, the first kStages - 1 tiles in flight
    for (int vv = 0; vv < kStages; ++vv)
        fetch_desc(vv);
    asm volatile("cp.async.wait_group 0;" ::: "memory");
    __syncwarp();
    int issued = 0;
    while (issued < known && issued < kStages - 1) {
        const int sidx = issued % kStages;
        if (lane == 0)
            issue_tile(t, ring[issued & (kDescRing - 1)], wsm + sidx * SL.bytes, SL, bar0 + 8 * sidx, false,
                       (first_warp && issued == 0) ? a.hold_tx : 0u);
        ++issued;
    }
    __syncwarp();

    int64_t big_first = 0;
    Best big_carry = best_none();
    Best big_priv = best_none();
    int failed_at = -1;
    int v = 0;
    for (; v < known; ++v) {
        // the copy of the next tile (its descriptor was requested one tile ago, or in the prologue),
        // then the request of the descriptor after it
        take_until(v + kStages + 1);
        if (issued < known) {
            asm volatile("cp.async.wait_group 0;" ::: "memory");
            __syncwarp();
            if (lane == 0) {
                const int sidx = issued % kStages;
                issue_tile(t, ring[issued & (kDescRing - 1)], wsm + sidx * SL.bytes, SL, bar0 + 8 * sidx, false);
            }
            ++issued;
            fetch_desc(issued);
        }
        const int slot = qh % kPersistQueue;
        const int round = q_item[slot] / NR;
        const TileDesc d = ring[v & (kDescRing - 1)];
        const int sidx = v % kStages;
        const uint32_t parity = (uint32_t)((v / kStages) & 1);
        if (!__all_sync(FULL, wait_stage(bar0 + 8 * sidx, parity, st.err, a.wait_ms))) {
            failed_at = v;
            break;
        }
        if (d.scenario != c.s || round != c.round) {
            // a new scenario or round: the arrival (in tiles) for the one left, then the wait for
            // this one's prices
            flush<RT, G>(c, lane);
            c.s = -1;
            if (!wait_version(st.ver, d.scenario, round, st.err, a.wait_ms, st.stats)) {
                failed_at = v;
                break;
            }
            c.round = round;
            enter_scenario<RT, G>(c, d.scenario, nullptr, lane);
        }
        if (!c.sp.skip) {
            ++c.ntiles;
            const StagePtrs ptrs = stage_ptrs_il(d, wsm + sidx * SL.bytes, SL, c.R);
            if (UNI && c.uniform_k >= 4)
                process_tile_uniform4<RT, G, F>(c, d, ptrs, lane);
            else if (UNI)
                process_tile_uniform<RT, G, F>(c, d, ptrs, lane, c.uniform_k, c.log2_k);
            else if (d.flags & TILE_BIG)
                process_tile_bigchunk<RT, G, F>(c, d, ptrs, big_first, big_priv, lane);
            else if ((d.flags & TILE_RUN) && tile_run_k(d.flags) >= 4)
                process_tile_run4<RT, G, F>(c, d, ptrs, lane, tile_run_k(d.flags));
            else if (d.flags & TILE_RUN)
                process_tile_uniform<RT, G, F>(c, d, ptrs, lane, tile_run_k(d.flags), tile_run_k(d.flags) >> 1);
        }
        __syncwarp();
        if (v + 1 == q_vs[slot] + q_len[slot])   // the end of an item
            ++qh;
    }
    asm volatile("cp.async.wait_group 0;" ::: "memory");
    if (failed_at < 0) {
        flush<RT, G>(c, lane);
    } else {
        // a wait gave up: wait (bounded) for every copy still in flight, then leave
        for (int vv = failed_at; vv < issued; ++vv)
            wait_stage(bar0 + 8 * (vv % kStages), (uint32_t)((vv / kStages) & 1), st.err, a.wait_ms);
    }
}

// Launch of the persistent pass (cooperative: every CTA co-resident).
template <int RT, int MODE, bool F>
struct PersistKernel {
    static const void *fn() { return reinterpret_cast<const void *>(&k_pass_persist<RT, MODE, F>); }
    static cudaError_t launch(int grid, int smem, cudaStream_t stream, const DevTable &t, const DevState &st,
                              const DevPlan &pl, const SolveArgs &a, int n_rounds)
    {
        cudaLaunchConfig_t cfg = {};
        cfg.gridDim = dim3((unsigned)grid);
        cfg.blockDim = dim3(kWarpsPerCta * 32);
        cfg.dynamicSmemBytes = (size_t)smem;
        cfg.stream = stream;
        cudaLaunchAttribute attr[1];
        attr[0].id = cudaLaunchAttributeCooperative;
        attr[0].val.cooperative = 1;
        cfg.attrs = attr;
        cfg.numAttrs = 1;
        return cudaLaunchKernelEx(&cfg, k_pass_persist<RT, MODE, F>, t, st, pl, a, n_rounds);
    }
};

// Resident CTAs per SM of both instantiations of K (the smaller), after setting their dynamic
// shared memory limit; 0 if either cannot run.
template <typename K>
int pass_kernels_ctas_per_sm(int smem)
{
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
}

}  // namespace

}  // namespace esp
