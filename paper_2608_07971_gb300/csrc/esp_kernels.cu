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
#include "esp_warp.cuh"

namespace esp {

namespace {

// ---------------------------------------------------------------------------------------------
// PTX helpers: mbarrier + 1-D bulk copy (TMA engine), sm_90+ forms that sm_103a accepts.

__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count)
{
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}

__device__ __forceinline__ void fence_barrier_init()
{
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint32_t bar, uint32_t bytes)
{
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes) : "memory");
}

// Waits on the phase of the given parity; the thread may sleep until the phase completes or about
// suspend_ns elapse, whichever is first.
__device__ __forceinline__ bool mbar_try_wait(uint32_t bar, uint32_t parity, uint32_t suspend_ns)
{
    uint32_t done;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2, %3;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(done)
        : "r"(bar), "r"(parity), "r"(suspend_ns)
        : "memory");
    return done != 0;
}

__device__ __forceinline__ void bulk_g2s(uint32_t dst, const void *src, uint32_t bytes, uint32_t bar)
{
    asm volatile(
        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(dst),
        "l"(src), "r"(bytes), "r"(bar)
        : "memory");
}

// Hint: bring [src, src + bytes) into L2 (16-byte aligned address and size).
__device__ __forceinline__ void prefetch_l2(const void *src, uint32_t bytes)
{
    asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(src), "r"(bytes) : "memory");
}

__device__ __forceinline__ void fence_proxy_async()
{
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

// Bounded wait on a stage barrier: sleeps until the copy lands (each attempt sleeps at most ~1 ms)
// and gives up after 4096 attempts (seconds), flags a timeout and returns false so the kernel can
// finish instead of hanging.
__device__ __forceinline__ bool wait_stage(uint32_t bar, uint32_t parity, unsigned int *err)
{
    for (uint32_t it = 0; it < kWaitPolls; ++it)
        if (mbar_try_wait(bar, parity, kWaitSuspendNs))
            return true;
    atomicOr(err, DEV_ERR_TIMEOUT);
    return false;
}


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
template <int RT, bool G>
__device__ __forceinline__ bool load_option(const WarpCtx<RT, G> &c, bool in_smem, const int32_t *units_s,
                                            const double *vals_s, const uint16_t *grp_s, int o, int64_t gfirst,
                                            int32_t *u, double &v, int &g)
{
    const int R = c.R;
    bool dup;
    g = 0;
    if (in_smem) {
        dup = load_units_smem<RT>(units_s + (size_t)o * R, u, R);
        v = vals_s[o];
        if (G)
            g = grp_s[o];
    } else {
        const int64_t og = gfirst + o;
        dup = load_units_global<RT>(c.t.units + og * R, u, R);
        v = __ldg(c.t.values + og);
        if (G)
            g = __ldg(c.t.group + og);
    }
    return dup;
}

// Exact resolution of one job whose screen was ambiguous. Survivors are the options with
// q <= thr (every option in exact mode), duplicates excluded (each has an earlier identical twin,
// so it can never be the lexicographic minimum); the answer is the survivors' minimum of
// (s, index). A survivor whose data equal those of the lowest-index survivor c0 (a duplicate the
// load-time marking did not cover) is skipped for the same reason, so only survivors that differ
// from c0 are rescored in fp64. q is recomputed with the same instructions as the screen.
// Returns the job-local index; s_out is set when has_s is true (always when need_s).
template <int RT, bool G>
__device__ void resolve_job(WarpCtx<RT, G> &c, int lane, bool in_smem, const int32_t *units_s, const double *vals_s,
                            const uint16_t *grp_s, int jstart, int jend, int64_t gfirst, float thr, bool need_s,
                            double &s_out, bool &has_s, int &local_out)
{
    const int R = c.R;
    int32_t u[Cols<RT>::N];
    double v;
    int g;
    int first = kIdxNone;
    for (int o = jstart + lane; o < jend; o += 32) {
        if (load_option<RT, G>(c, in_smem, units_s, vals_s, grp_s, o, gfirst, u, v, g))
            continue;
        if (c.sp.exact || screen_score<RT, G>(u, v, g, c.sp, R, c.rg) <= thr) {
            first = o;
            break;
        }
    }
    first = __reduce_min_sync(FULL, first);
    int32_t u0[Cols<RT>::N];
    double v0;
    int g0;
    load_option<RT, G>(c, in_smem, units_s, vals_s, grp_s, first, gfirst, u0, v0, g0);

    long long best_key = 0x7fffffffffffffffLL;
    int best_i = kIdxNone;
    bool distinct = false;
    for (int o = jstart + lane; o < jend; o += 32) {
        if (o <= first)
            continue;
        if (load_option<RT, G>(c, in_smem, units_s, vals_s, grp_s, o, gfirst, u, v, g))
            continue;
        if (!(c.sp.exact || screen_score<RT, G>(u, v, g, c.sp, R, c.rg) <= thr))
            continue;
        bool same = (__double_as_longlong(v) == __double_as_longlong(v0)) && (g == g0);
#pragma unroll
        for (int r = 0; r < Cols<RT>::N; ++r)
            if (RT != 0 || r < R)
                same &= (u[r] == u0[r]);
        if (same)
            continue;
        distinct = true;
        const long long k = order_key(exact_score<RT, G>(u, v, g, c.sp, R, c.rg));
        if (k < best_key || (k == best_key && o < best_i)) {
            best_key = k;
            best_i = o;
        }
    }
    if (!__any_sync(FULL, distinct)) {
        local_out = first - jstart;
        has_s = need_s;
        if (need_s)
            s_out = exact_score<RT, G>(u0, v0, g0, c.sp, R, c.rg);
        return;
    }
    if (lane == 0) {
        const long long k0 = order_key(exact_score<RT, G>(u0, v0, g0, c.sp, R, c.rg));
        if (k0 < best_key || (k0 == best_key && first < best_i)) {
            best_key = k0;
            best_i = first;
        }
    }
#pragma unroll
    for (int d = 16; d >= 1; d >>= 1) {
        const long long ok = __shfl_xor_sync(FULL, best_key, d);
        const int oi = __shfl_xor_sync(FULL, best_i, d);
        if (ok < best_key || (ok == best_key && oi < best_i)) {
            best_key = ok;
            best_i = oi;
        }
    }
    local_out = best_i - jstart;
    s_out = key_value(best_key);
    has_s = true;
}

// Resolves, one after the other, the ambiguous jobs whose closing lanes are set in amask, and records
// each winner (lane 0). big: the job is chunked and read from global memory.
template <int RT, bool G>
__device__ __forceinline__ void resolve_row(WarpCtx<RT, G> &c, int lane, uint32_t amask, bool big,
                                            const int32_t *units_s, const double *vals_s, const uint16_t *grp_s,
                                            int jstart, int jend, float thr, int64_t job, int64_t big_first)
{
    while (amask) {
        const int cl = __ffs(amask) - 1;
        amask &= amask - 1;
        const int js = __shfl_sync(FULL, jstart, cl);
        const int je = __shfl_sync(FULL, jend, cl);
        const float th = __shfl_sync(FULL, thr, cl);
        const long long jb = __shfl_sync(FULL, (long long)job, cl);
        double s_w = 0.0;
        bool has_s = false;
        int li;
        resolve_job<RT, G>(c, lane, !big, units_s, vals_s, grp_s, js, je, big ? big_first : 0, th, c.want_min,
                           s_w, has_s, li);
        if (lane == 0) {
            atomicAdd(c.st.stats, 1ull);
            int32_t uw[Cols<RT>::N];
            double vw;
            int gw;
            load_option<RT, G>(c, !big, units_s, vals_s, grp_s, js + li, big ? big_first : 0, uw, vw, gw);
            take_winner<RT, G>(c, jb, li, uw, vw, gw, has_s, s_w);
        }
    }
}

// Stage pointers of one tile (the bulk copies start at the 16-byte boundary below the data).
struct StagePtrs {
    const int32_t *units;
    const double *vals;
    const uint16_t *grp;
    const long long *off;
};

__device__ __forceinline__ StagePtrs stage_ptrs(const TileDesc &d, const unsigned char *stage, const StageLayout &SL,
                                                int R)
{
    StagePtrs p;
    p.units = reinterpret_cast<const int32_t *>(stage + SL.units + (int)((d.opt_begin * R * 4) & 15));
    p.vals = reinterpret_cast<const double *>(stage + SL.vals + (int)((d.opt_begin * 8) & 15));
    p.grp = reinterpret_cast<const uint16_t *>(stage + SL.grp + (int)((d.opt_begin * 2) & 15));
    p.off = reinterpret_cast<const long long *>(stage + SL.off + (int)((d.job_begin * 8) & 15));
    return p;
}

// Tile of a table whose jobs all have K = uniform_k options (a power of two <= 32). Tiles start at
// job boundaries, so each aligned group of K lanes of a row is one job: a log2(K)-step xor
// butterfly gives every lane of the group the smallest and second-smallest screen value; when the
// job is unambiguous the unique lane holding the smallest value is the winner and records it from
// its own registers.
template <int RT, bool G>
__device__ void process_tile_uniform(WarpCtx<RT, G> &c, const TileDesc &d, const StagePtrs &sp, int lane, int K,
                                     int log2_k)
{
    const int R = c.R;
    const int n = d.n_opt;
    for (int b = 0; b < n; b += 32) {
        const int i = b + lane;
        const bool valid = i < n;
        int32_t u[Cols<RT>::N];
        double v = 0.0;
        int g = 0;
        float q = INFINITY;
        if (valid) {
            const bool dup = load_units_smem<RT>(sp.units + (size_t)i * R, u, R);
            v = sp.vals[i];
            if (G)
                g = sp.grp[i];
            if (!dup)
                q = screen_score<RT, G>(u, v, g, c.sp, R, c.rg);
        }
        float m1 = q, m2 = INFINITY;
        for (int dd = 1; dd < K; dd <<= 1) {
            const float o1 = __shfl_xor_sync(FULL, m1, dd);
            const float o2 = __shfl_xor_sync(FULL, m2, dd);
            m2 = fminf(fminf(m2, o2), fmaxf(m1, o1));
            m1 = fminf(m1, o1);
        }
        const float thr = __fadd_ru(m1, c.sp.e2);
        const bool amb = c.sp.exact || !(m2 > thr);
        const int64_t job = d.job_begin + (i >> log2_k);
        if (valid && !amb && q == m1)
            take_winner<RT, G>(c, job, i & (K - 1), u, v, g, false, 0.0);
        const uint32_t amask = __ballot_sync(FULL, valid && amb && (i & (K - 1)) == 0);
        if (amask)
            resolve_row<RT, G>(c, lane, amask, false, sp.units, sp.vals, sp.grp, i, i + K, thr, job, 0);
    }
}

// Units of the 4 consecutive options starting at p (16-byte aligned): six, four or eight 16-byte
// shared loads for R = 6, 4, 8. Duplicate marks are removed and returned in dup[].
template <int RT>
__device__ __forceinline__ void load_units4_smem(const int32_t *p, int32_t (*u)[Cols<RT>::N], bool *dup, int R)
{
    if constexpr (RT == 4 || RT == 6 || RT == 8) {
        constexpr int W = RT;
        int32_t raw[4 * W];
        const int4 *q4 = reinterpret_cast<const int4 *>(p);
#pragma unroll
        for (int k = 0; k < W; ++k) {
            const int4 x = q4[k];
            raw[4 * k] = x.x; raw[4 * k + 1] = x.y; raw[4 * k + 2] = x.z; raw[4 * k + 3] = x.w;
        }
#pragma unroll
        for (int o = 0; o < 4; ++o)
#pragma unroll
            for (int r = 0; r < W; ++r)
                u[o][r] = raw[o * W + r];
    } else {
#pragma unroll
        for (int o = 0; o < 4; ++o)
#pragma unroll
            for (int r = 0; r < Cols<RT>::N; ++r)
                u[o][r] = (r < R) ? p[o * R + r] : 0;
    }
#pragma unroll
    for (int o = 0; o < 4; ++o) {
        dup[o] = u[o][0] < 0;
        u[o][0] &= 0x7fffffff;
    }
}

// Exact resolution inside a row of the four-options-per-lane layout: every lane of an ambiguous job
// rescores in fp64 its own survivors among the four options it screened (q <= thr; every option
// but the duplicates in exact mode), then an xor butterfly over the job's L lanes keeps the
// lexicographic minimum of (s, job-local index), and the lane holding that option records it.
// The options are still in the stage, so no option is read twice from memory. base: tile-local
// index of the lane's first option; loc0: its job-local index; lamb: the lane's job is ambiguous.
template <int RT, bool G>
__device__ __forceinline__ void resolve4_in_row(WarpCtx<RT, G> &c, const StagePtrs &sp, bool lamb, const float *q,
                                                uint32_t dupmask, float thr, int base, int loc0, int64_t job, int L)
{
    long long key = 0x7fffffffffffffffLL;
    int bi = kIdxNone;
    if (lamb) {
#pragma unroll
        for (int o = 0; o < 4; ++o) {
            const bool cand = c.sp.exact ? !((dupmask >> o) & 1u) : (q[o] <= thr);
            if (!cand)
                continue;
            int32_t u[Cols<RT>::N];
            load_units_smem<RT>(sp.units + (size_t)(base + o) * c.R, u, c.R);
            const long long k = order_key(exact_score<RT, G>(u, sp.vals[base + o], 0, c.sp, c.R, c.rg));
            if (k < key) {
                key = k;
                bi = loc0 + o;
            }
        }
    }
    for (int dd = 1; dd < L; dd <<= 1) {
        const long long ok = __shfl_xor_sync(FULL, key, dd);
        const int oi = __shfl_xor_sync(FULL, bi, dd);
        if (ok < key || (ok == key && oi < bi)) {
            key = ok;
            bi = oi;
        }
    }
    if (lamb && bi >= loc0 && bi < loc0 + 4) {
        const int i = base + (bi - loc0);
        int32_t uw[Cols<RT>::N];
        load_units_smem<RT>(sp.units + (size_t)i * c.R, uw, c.R);
        take_winner<RT, G>(c, job, bi, uw, sp.vals[i], 0, true, key_value(key));
        atomicAdd(c.st.stats, 1ull);
    }
}

// Tile of a table whose jobs all have K options, K in {4, 8, 16, 32}. Each lane evaluates 4
// consecutive options of one job (a tile row block is 128 options), keeps their smallest and
// second-smallest screen values, and a log2(K / 4)-step xor butterfly over the job's K / 4 lanes
// completes the job. An unambiguous job's winner is the unique option holding the smallest value.
template <int RT, bool G>
__device__ void process_tile_uniform4(WarpCtx<RT, G> &c, const TileDesc &d, const StagePtrs &sp, int lane)
{
    const int R = c.R;
    const int n = d.n_opt;
    const int K = c.uniform_k;
    const int KL = K >> 2;                  // lanes per job
    for (int b = 0; b < n; b += 128) {
        const int base = b + 4 * lane;
        const bool valid = base < n;        // n is a multiple of K, hence of 4
        float q[4] = {INFINITY, INFINITY, INFINITY, INFINITY};
        uint32_t dupmask = 0;
        if (valid) {
            int32_t u[4][Cols<RT>::N];
            bool dup[4];
            load_units4_smem<RT>(sp.units + (size_t)base * R, u, dup, R);
            const double2 va = reinterpret_cast<const double2 *>(sp.vals + base)[0];
            const double2 vb = reinterpret_cast<const double2 *>(sp.vals + base)[1];
            const double v[4] = {va.x, va.y, vb.x, vb.y};
#pragma unroll
            for (int o = 0; o < 4; ++o) {
                dupmask |= dup[o] ? (1u << o) : 0u;
                if (!dup[o])
                    q[o] = screen_score<RT, G>(u[o], v[o], 0, c.sp, R, c.rg);
            }
        }
        // smallest and second smallest of the lane's four values
        float a0 = fminf(q[0], q[1]), a1 = fmaxf(q[0], q[1]);
        float b0 = fminf(q[2], q[3]), b1 = fmaxf(q[2], q[3]);
        float m1 = fminf(a0, b0);
        float m2 = fminf(fmaxf(a0, b0), fminf(a1, b1));
        for (int dd = 1; dd < KL; dd <<= 1) {
            const float o1 = __shfl_xor_sync(FULL, m1, dd);
            const float o2 = __shfl_xor_sync(FULL, m2, dd);
            m2 = fminf(fminf(m2, o2), fmaxf(m1, o1));
            m1 = fminf(m1, o1);
        }
        const float thr = __fadd_ru(m1, c.sp.e2);
        const bool amb = c.sp.exact || !(m2 > thr);
        if (valid && !amb) {
            int w = -1;
#pragma unroll
            for (int o = 3; o >= 0; --o)
                if (q[o] == m1)
                    w = o;
            if (w >= 0) {
                const int i = base + w;
                int32_t uw[Cols<RT>::N];
                load_units_smem<RT>(sp.units + (size_t)i * R, uw, R);
                take_winner<RT, G>(c, d.job_begin + (i >> c.log2_k), i & (K - 1), uw, sp.vals[i], 0, false, 0.0);
            }
        }
        const bool lamb = valid && amb;
        if (__any_sync(FULL, lamb))
            resolve4_in_row<RT, G>(c, sp, lamb, q, dupmask, thr, base, base & (K - 1),
                                   d.job_begin + (base >> c.log2_k), KL);
    }
}

// Tile of a run of the sorted layout whose jobs all have K = 4m options (m <= 32). Every job owns
// L = 2^ceil(log2 m) lanes; lane `sub` of a job evaluates its options 4 sub .. 4 sub + 3 (16-byte
// shared loads: the run starts on a 4-option boundary), lanes with sub >= m idle, and a
// log2(L)-step xor butterfly completes the job as in the uniform path.
template <int RT, bool G>
__device__ void process_tile_run4(WarpCtx<RT, G> &c, const TileDesc &d, const StagePtrs &sp, int lane, int K)
{
    const int R = c.R;
    const int m = K >> 2;
    const int log2L = 32 - __clz(m - 1);
    const int L = 1 << log2L;
    const int jobs_per_row = 32 >> log2L;
    const int jslot = lane >> log2L, sub = lane & (L - 1);
    const int n_job = d.n_job;
    for (int jb = 0; jb < n_job; jb += jobs_per_row) {
        const int jl = jb + jslot;
        const bool valid = jl < n_job && sub < m;
        const int base = jl * K + 4 * sub;
        float q[4] = {INFINITY, INFINITY, INFINITY, INFINITY};
        uint32_t dupmask = 0;
        if (valid) {
            int32_t u[4][Cols<RT>::N];
            bool dup[4];
            load_units4_smem<RT>(sp.units + (size_t)base * R, u, dup, R);
            const double2 va = reinterpret_cast<const double2 *>(sp.vals + base)[0];
            const double2 vb = reinterpret_cast<const double2 *>(sp.vals + base)[1];
            const double v[4] = {va.x, va.y, vb.x, vb.y};
#pragma unroll
            for (int o = 0; o < 4; ++o) {
                dupmask |= dup[o] ? (1u << o) : 0u;
                if (!dup[o])
                    q[o] = screen_score<RT, G>(u[o], v[o], 0, c.sp, R, c.rg);
            }
        }
        float a0 = fminf(q[0], q[1]), a1 = fmaxf(q[0], q[1]);
        float b0 = fminf(q[2], q[3]), b1 = fmaxf(q[2], q[3]);
        float m1 = fminf(a0, b0);
        float m2 = fminf(fmaxf(a0, b0), fminf(a1, b1));
        for (int dd = 1; dd < L; dd <<= 1) {
            const float o1 = __shfl_xor_sync(FULL, m1, dd);
            const float o2 = __shfl_xor_sync(FULL, m2, dd);
            m2 = fminf(fminf(m2, o2), fmaxf(m1, o1));
            m1 = fminf(m1, o1);
        }
        const float thr = __fadd_ru(m1, c.sp.e2);
        const bool amb = c.sp.exact || !(m2 > thr);
        const int64_t job = d.job_begin + jl;
        if (valid && !amb) {
            int w = -1;
#pragma unroll
            for (int o = 3; o >= 0; --o)
                if (q[o] == m1)
                    w = o;
            if (w >= 0) {
                const int i = base + w;
                int32_t uw[Cols<RT>::N];
                load_units_smem<RT>(sp.units + (size_t)i * R, uw, R);
                take_winner<RT, G>(c, job, 4 * sub + w, uw, sp.vals[i], 0, false, 0.0);
            }
        }
        const bool lamb = valid && amb;
        if (__any_sync(FULL, lamb))
            resolve4_in_row<RT, G>(c, sp, lamb, q, dupmask, thr, base, 4 * sub, job, L);
    }
}

// Tile of a general table (any job sizes). Rows of 32 options are reduced by a segmented scan:
// heads (first options) and ends (last options) of jobs in the row come from the staged job
// offsets; a job continuing from the previous row enters as a carry; rows entirely inside one job
// only fold per lane. A job larger than a tile arrives as consecutive chunk tiles of this warp
// (big_first / big_carry carry its state across them) and is resolved from global memory.
template <int RT, bool G>
__device__ void process_tile_general(WarpCtx<RT, G> &c, const TileDesc &d, const StagePtrs &sp, int64_t &big_first,
                                     Best &big_carry, int lane)
{
    const int R = c.R;
    const int n = d.n_opt;
    const bool big = (d.flags & TILE_BIG) != 0;
    int chunk_base = 0;
    Best carry = best_none();
    if (big) {
        if (d.flags & TILE_BIG_FIRST) {
            big_first = d.opt_begin;
            big_carry = best_none();
        }
        chunk_base = (int)(d.opt_begin - big_first);
        carry = big_carry;
    }
    Best priv = best_none();
    bool priv_dirty = false;
    int open_start = 0;      // tile-local start of the job open at the start of the row
    int wp = 0;              // first job of the tile not yet closed
    const int n_job = d.n_job;

    for (int b = 0; b < n; b += 32) {
        const int i = b + lane;
        const bool valid = i < n;
        int32_t u[Cols<RT>::N];
        float q = INFINITY;
        if (valid) {
            const bool dup = load_units_smem<RT>(sp.units + (size_t)i * R, u, R);
            const double v = sp.vals[i];
            const int g = G ? (int)sp.grp[i] : 0;
            if (!dup)
                q = screen_score<RT, G>(u, v, g, c.sp, R, c.rg);
        }

        // heads (first option of a job) and ends (last option of a job) in this row
        uint32_t H, E;
        if (!big) {
            const int k0 = wp + lane;
            const int sa = (k0 < n_job) ? (int)(sp.off[k0] - d.opt_begin) : 0x7fffffff;
            const int sb = (k0 + 1 < n_job) ? (int)(sp.off[k0 + 1] - d.opt_begin) : (k0 + 1 == n_job ? n : 0x7fffffff);
            const int hb = sa - b, eb = sb - 1 - b;
            H = __reduce_or_sync(FULL, (hb >= 0 && hb < 32) ? (1u << hb) : 0u);
            E = __reduce_or_sync(FULL, (eb >= 0 && eb < 32) ? (1u << eb) : 0u);
        } else {
            H = ((d.flags & TILE_BIG_FIRST) && b == 0) ? 1u : 0u;
            const int eb = n - 1 - b;
            E = ((d.flags & TILE_BIG_LAST) && eb >= 0 && eb < 32) ? (1u << eb) : 0u;
        }

        Best x = valid ? Best{q, i + chunk_base, INFINITY} : best_none();
        if (H == 0u && E == 0u) {    // the whole row lies inside the open job: fold per lane
            priv = combine(priv, x);
            priv_dirty = true;
            continue;
        }
        if (priv_dirty) {
            carry = combine(carry, allreduce_best(priv));
            priv = best_none();
            priv_dirty = false;
        }
        // segmented inclusive scan; lanes before the first head continue the open job (carry)
        const uint32_t le = (lane == 31) ? FULL : ((2u << lane) - 1u);
        const int seg_lo = 31 - __clz(H & le);
        if (H != FULL) {
#pragma unroll
            for (int dd = 1; dd < 32; dd <<= 1) {
                const Best o = shfl_up_best(x, dd);
                if (lane >= dd && lane - dd >= seg_lo)
                    x = combine(o, x);
            }
        }
        if (seg_lo < 0)
            x = combine(carry, x);

        const bool closing = (E >> lane) & 1u;
        const uint32_t lt = (1u << lane) - 1u;
        const int jstart = big ? 0 : ((seg_lo >= 0) ? (b + seg_lo) : open_start);
        const int64_t job = big ? d.job_begin : (d.job_begin + wp + __popc(E & lt));
        const int jend = big ? (chunk_base + i + 1) : (i + 1);

        // next row's open job
        const Best last = shfl_best(x, 31);
        const int last_start = __shfl_sync(FULL, jstart, 31);
        if ((E >> 31) & 1u) {
            carry = best_none();
        } else {
            carry = last;
            open_start = last_start;
        }
        if (!big)
            wp += __popc(E);

        // unambiguous closings finish here; ambiguous ones are resolved exactly by the warp
        const float thr = __fadd_ru(x.m1, c.sp.e2);
        const bool amb = closing && (c.sp.exact || !(x.m2 > thr));
        if (closing && !amb) {
            const int li = big ? x.idx : (x.idx - jstart);
            int32_t uw[Cols<RT>::N];
            double vw;
            int gw;
            load_option<RT, G>(c, !big, sp.units, sp.vals, sp.grp, big ? x.idx : x.idx, big ? big_first : 0, uw, vw,
                               gw);
            take_winner<RT, G>(c, job, li, uw, vw, gw, false, 0.0);
        }
        const uint32_t amask = __ballot_sync(FULL, amb);
        if (amask)
            resolve_row<RT, G>(c, lane, amask, big, sp.units, sp.vals, sp.grp, jstart, jend, thr, job, big_first);
    }
    if (big) {
        if (priv_dirty)
            carry = combine(carry, allreduce_best(priv));
        big_carry = carry;
    }
}

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
// needed. Each lane folds the options it owns (lane-strided: conflict-free shared loads) into a
// lane-private state carried across the job's chunks; the job's last chunk reduces the states across
// the warp once and records the winner (exact resolution from global memory when ambiguous).
template <int RT, bool G>
__device__ void process_tile_bigchunk(WarpCtx<RT, G> &c, const TileDesc &d, const StagePtrs &sp, int64_t &big_first,
                                      Best &big_priv, int lane)
{
    const int R = c.R;
    const int n = d.n_opt;
    if (d.flags & TILE_BIG_FIRST) {
        big_first = d.opt_begin;
        big_priv = best_none();
    }
    const int chunk_base = (int)(d.opt_begin - big_first);
#if ESP_BIGCHUNK4
    // four options per step (lane, lane + 32, lane + 64, lane + 96): their loads and screens are
    // independent; the lane's state then takes them in increasing index order (strict <, so the
    // lowest index keeps a tie)
    for (int i0 = lane; i0 < n; i0 += 128) {
        float q[4];
#pragma unroll
        for (int o = 0; o < 4; ++o) {
            const int i = i0 + 32 * o;
            q[o] = INFINITY;
            if (i < n) {
                int32_t u[Cols<RT>::N];
                const bool dup = load_units_smem<RT>(sp.units + (size_t)i * R, u, R);
                const double v = sp.vals[i];
                const int g = G ? (int)sp.grp[i] : 0;
                if (!dup)
                    q[o] = screen_score<RT, G>(u, v, g, c.sp, R, c.rg);
            }
        }
#pragma unroll
        for (int o = 0; o < 4; ++o) {
            const bool better = q[o] < big_priv.m1;
            big_priv.m2 = better ? big_priv.m1 : fminf(big_priv.m2, q[o]);
            big_priv.idx = better ? chunk_base + i0 + 32 * o : big_priv.idx;
            big_priv.m1 = fminf(big_priv.m1, q[o]);
        }
    }
#else
    for (int i = lane; i < n; i += 32) {
        int32_t u[Cols<RT>::N];
        const bool dup = load_units_smem<RT>(sp.units + (size_t)i * R, u, R);
        const double v = sp.vals[i];
        const int g = G ? (int)sp.grp[i] : 0;
        const float q = dup ? INFINITY : screen_score<RT, G>(u, v, g, c.sp, R, c.rg);
        big_priv = combine(big_priv, Best{q, dup ? kIdxNone : chunk_base + i, INFINITY});
    }
#endif
    if (!(d.flags & TILE_BIG_LAST))
        return;
    const Best x = allreduce_best(big_priv);
    const float thr = __fadd_ru(x.m1, c.sp.e2);
    const bool amb = c.sp.exact || !(x.m2 > thr);
    const int K = chunk_base + n;
    if (!amb) {
        if (lane == 0) {
            int32_t uw[Cols<RT>::N];
            double vw;
            int gw;
            load_option<RT, G>(c, false, sp.units, sp.vals, sp.grp, x.idx, big_first, uw, vw, gw);
            take_winner<RT, G>(c, d.job_begin, x.idx, uw, vw, gw, false, 0.0);
        }
    } else if (!c.sp.exact && !__any_sync(FULL, big_priv.m2 <= thr)) {
        // every lane holds at most one survivor (q <= thr), its own smallest: those are rescored in
        // fp64 from global memory, one per lane, and the warp keeps the minimum of (s, index)
        long long key = 0x7fffffffffffffffLL;
        int bi = kIdxNone;
        if (big_priv.m1 <= thr) {
            int32_t u[Cols<RT>::N];
            double v;
            int g;
            load_option<RT, G>(c, false, sp.units, sp.vals, sp.grp, big_priv.idx, big_first, u, v, g);
            key = order_key(exact_score<RT, G>(u, v, g, c.sp, c.R, c.rg));
            bi = big_priv.idx;
        }
#pragma unroll
        for (int dd = 16; dd >= 1; dd >>= 1) {
            const long long ok = __shfl_xor_sync(FULL, key, dd);
            const int oi = __shfl_xor_sync(FULL, bi, dd);
            if (ok < key || (ok == key && oi < bi)) {
                key = ok;
                bi = oi;
            }
        }
        if (lane == 0) {
            int32_t uw[Cols<RT>::N];
            double vw;
            int gw;
            load_option<RT, G>(c, false, sp.units, sp.vals, sp.grp, bi, big_first, uw, vw, gw);
            take_winner<RT, G>(c, d.job_begin, bi, uw, vw, gw, true, key_value(key));
            atomicAdd(c.st.stats, 1ull);
        }
    } else {
        resolve_row<RT, G>(c, lane, 1u, true, sp.units, sp.vals, sp.grp, 0, K, thr, d.job_begin, big_first);
    }
}

// Issues the bulk copies of tile d into a stage; lane 0 only (issuing the copies from several lanes
// at once measured slower). Uniform tables and runs of the sorted layout need no job offsets.
__device__ __forceinline__ void issue_tile(const DevTable &t, const TileDesc &d, unsigned char *stage,
                                           const StageLayout &SL, uint32_t bar, bool need_offsets)
{
    const int R = t.R;
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
    mbar_arrive_expect_tx(bar, total);
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
template <int RT, bool UNI>
constexpr int pass_min_ctas()
{
    return UNI ? ((RT == 4 || RT == 6) ? kMinCtasPerSmNarrow : kMinCtasPerSm) : kMinCtasPerSmGeneral;
}

template <int RT, bool G, bool UNI, bool PLAIN>
__global__ void __launch_bounds__(kWarpsPerCta * 32, pass_min_ctas<RT, UNI>()) k_pass(DevTable t, DevState st, DevPlan pl,
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

    const WarpSmem WS = warp_smem(pl.tile_opt, t.R, G, t.P, !UNI);
    const StageLayout SL = stage_layout(pl.tile_opt, t.R, G, !UNI);
    unsigned char *wsm = smem + (size_t)wid * WS.bytes;
    float *p32s = reinterpret_cast<float *>(wsm + WS.p32);
    const uint32_t bar0 = smem_u32(wsm + WS.bars);
    const bool need_offsets = !UNI;

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
                       need_offsets);
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
        if (!__all_sync(FULL, wait_stage(bar0 + 8 * sidx, parity, st.err))) {   // uniform decision
            failed_at = k;
            break;
        }
        if (d.scenario != c.s)
            enter_scenario<RT, G>(c, d.scenario, p32s, lane);
        if (!c.sp.skip) {
            const StagePtrs ptrs = stage_ptrs(d, wsm + sidx * SL.bytes, SL, c.R);
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
            else
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
            wait_stage(bar0 + 8 * sidx, (uint32_t)(((k - k_begin) / kStages) & 1), st.err);
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
template <int RT, bool G, bool UNI>
struct PassKernels {
    static const void *plain() { return reinterpret_cast<const void *>(&k_pass<RT, G, UNI, true>); }
    static const void *other() { return reinterpret_cast<const void *>(&k_pass<RT, G, UNI, false>); }
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
            cudaLaunchKernelEx(&cfg, k_pass<RT, G, UNI, true>, t, st, pl, a, round, kind);
        else
            cudaLaunchKernelEx(&cfg, k_pass<RT, G, UNI, false>, t, st, pl, a, round, kind);
    }
};

// Calls f.template operator()<RT, G, UNI>() for the instantiation that serves this table shape.
template <typename F>
auto dispatch_shape(int R, bool grouped, bool uni, F &&f)
{
    if (grouped) {
        switch (R) {
        case 4: return f(PassKernels<4, true, false>());
        case 6: return f(PassKernels<6, true, false>());
        case 8: return f(PassKernels<8, true, false>());
        default: return f(PassKernels<0, true, false>());
        }
    }
    if (uni) {
        switch (R) {
        case 4: return f(PassKernels<4, false, true>());
        case 6: return f(PassKernels<6, false, true>());
        case 8: return f(PassKernels<8, false, true>());
        default: return f(PassKernels<0, false, true>());
        }
    }
    switch (R) {
    case 4: return f(PassKernels<4, false, false>());
    case 6: return f(PassKernels<6, false, false>());
    case 8: return f(PassKernels<8, false, false>());
    default: return f(PassKernels<0, false, false>());
    }
}

}  // namespace

int pass_smem_bytes(int R, bool grouped, bool uniform, int P, int tile_opt)
{
    return kWarpsPerCta * warp_smem(tile_opt, R, grouped, P, !uniform).bytes;
}

int pass_ctas_per_sm(int R, bool grouped, bool uniform, int P, int tile_opt)
{
    const int smem = pass_smem_bytes(R, grouped, uniform && !grouped, P, tile_opt);
    return dispatch_shape(R, grouped, uniform && !grouped, [&](auto k) -> int {
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
    const int smem = pass_smem_bytes(t.R, grouped, pl.uniform_k > 0, t.P, pl.tile_opt);
    const bool plain = kind == PASS_ROUND && st.hash_trace == nullptr && st.dual_trace == nullptr;
    dispatch_shape(t.R, grouped, pl.uniform_k > 0, [&](auto k) -> int {
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
