// Tile evaluation of the ESP best response (Sec. 3.2.2; Eq. esp_score without Gamma) for the
// evaluation-pass kernels: a warp scores the options of one staged tile with the fp32 screen,
// completes each job's (m1, index, m2) by shuffles, records unambiguous winners, and resolves
// ambiguous jobs exactly in fp64 (from the stage, or from global memory for chunked jobs).
#pragma once

#include <cmath>
#include <cstdint>
#include <cuda_runtime.h>

#include "esp_device.cuh"
#include "esp_kernels.h"
#include "esp_warp.cuh"

namespace esp {

namespace {

template <int RT, bool G, bool F>
__device__ __forceinline__ bool load_option(const WarpCtx<RT, G> &c, bool in_smem, const int32_t *units_s,
                                            const double *vals_s, const uint16_t *grp_s, int o, int64_t gfirst,
                                            int32_t *u, double &v, int &g)
{
    const int R = c.R;
    bool dup;
    g = 0;
    if (in_smem) {
        dup = load_units_stage<RT, F>(units_s + (size_t)o * R, u, R);
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
template <int RT, bool G, bool F>
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
        if (load_option<RT, G, F>(c, in_smem, units_s, vals_s, grp_s, o, gfirst, u, v, g))
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
    load_option<RT, G, F>(c, in_smem, units_s, vals_s, grp_s, first, gfirst, u0, v0, g0);

    long long best_key = 0x7fffffffffffffffLL;
    int best_i = kIdxNone;
    bool distinct = false;
    for (int o = jstart + lane; o < jend; o += 32) {
        if (o <= first)
            continue;
        if (load_option<RT, G, F>(c, in_smem, units_s, vals_s, grp_s, o, gfirst, u, v, g))
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
template <int RT, bool G, bool F>
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
        resolve_job<RT, G, F>(c, lane, !big, units_s, vals_s, grp_s, js, je, big ? big_first : 0, th, c.want_min,
                           s_w, has_s, li);
        if (lane == 0) {
            atomicAdd(c.st.stats, 1ull);
            int32_t uw[Cols<RT>::N];
            double vw;
            int gw;
            load_option<RT, G, F>(c, !big, units_s, vals_s, grp_s, js + li, big ? big_first : 0, uw, vw, gw);
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

// Stage pointers of one tile copied from the tile-interleaved table (DevTable::il): its units at the
// start of the stage's units region, its values right after them.
__device__ __forceinline__ StagePtrs stage_ptrs_il(const TileDesc &d, const unsigned char *stage,
                                                   const StageLayout &SL, int R)
{
    StagePtrs p;
    p.units = reinterpret_cast<const int32_t *>(stage + SL.units);
    p.vals = reinterpret_cast<const double *>(stage + SL.units + (size_t)d.n_opt * R * 4);
    p.grp = nullptr;
    p.off = nullptr;
    return p;
}

// Tile of a table whose jobs all have K = uniform_k options (a power of two <= 32). Tiles start at
// job boundaries, so each aligned group of K lanes of a row is one job: a log2(K)-step xor
// butterfly gives every lane of the group the smallest and second-smallest screen value; when the
// job is unambiguous the unique lane holding the smallest value is the winner and records it from
// its own registers.
template <int RT, bool G, bool F>
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
                q = screen_score_st<RT, G, F>(u, v, g, c.sp, R, c.rg);
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
        if (valid && !amb && q == m1) {
            stage_units_to_int<RT, F>(u, R);
            take_winner<RT, G>(c, job, i & (K - 1), u, v, g, false, 0.0);
        }
        const uint32_t amask = __ballot_sync(FULL, valid && amb && (i & (K - 1)) == 0);
        if (amask)
            resolve_row<RT, G, F>(c, lane, amask, false, sp.units, sp.vals, sp.grp, i, i + K, thr, job, 0);
    }
}

// Half-swap of a lane's four options (R = 6 only). A lane's 4 options span 96 bytes, so in each
// quarter-warp phase of a 16-byte shared load lanes l and l + 4 start in the same bank (96 bytes is
// 24 banks; four such strides wrap the 32 banks): a two-way conflict on every load. A lane whose
// group of four options has (group >> 2) odd reads the second half of its group (options 2, 3:
// 48 bytes = 12 banks further) first, which moves its 16-byte window off the other lanes' windows
// for every pair of the phase; its register slot s then holds option s ^ 2. The same swap of the two
// 16-byte value halves removes the two-way conflict of the value loads (32-byte lane stride).
// `opt0` is the tile-local index of the lane's first option (a multiple of 4).
template <int RT>
__device__ __forceinline__ int half_swap(int opt0)
{
    return RT == 6 ? (opt0 >> 4) & 1 : 0;
}

// Units of the 4 consecutive options starting at p (16-byte aligned): six, four or eight 16-byte
// shared loads for R = 6, 4, 8. Duplicate marks are removed and returned in dup[]. With rot = 1
// (R = 6, half_swap) slot s receives option s ^ 2.
template <int RT>
__device__ __forceinline__ void load_units4_smem(const int32_t *p, int32_t (*u)[Cols<RT>::N], bool *dup, int R,
                                                 int rot = 0)
{
    if constexpr (RT == 6) {
        int32_t raw[24];
        const int4 *q4 = reinterpret_cast<const int4 *>(p);
        const int4 *pa = q4 + 3 * rot, *pb = q4 + (3 - 3 * rot);
#pragma unroll
        for (int k = 0; k < 3; ++k) {
            const int4 x = pa[k];
            raw[4 * k] = x.x; raw[4 * k + 1] = x.y; raw[4 * k + 2] = x.z; raw[4 * k + 3] = x.w;
            const int4 y = pb[k];
            raw[12 + 4 * k] = y.x; raw[12 + 4 * k + 1] = y.y; raw[12 + 4 * k + 2] = y.z; raw[12 + 4 * k + 3] = y.w;
        }
#pragma unroll
        for (int o = 0; o < 4; ++o)
#pragma unroll
            for (int r = 0; r < 6; ++r)
                u[o][r] = raw[o * 6 + r];
    } else if constexpr (RT == 4 || RT == 8) {
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
template <int RT, bool G, bool F>
__device__ __forceinline__ void resolve4_in_row(WarpCtx<RT, G> &c, const StagePtrs &sp, bool lamb, const float *q,
                                                uint32_t dupmask, float thr, int base, int loc0, int64_t job, int L,
                                                int rot)
{
    long long key = 0x7fffffffffffffffLL;
    int bi = kIdxNone;
    if (lamb) {
#pragma unroll
        for (int s = 0; s < 4; ++s) {   // slot s holds option s ^ (2 rot)
            const bool cand = c.sp.exact ? !((dupmask >> s) & 1u) : (q[s] <= thr);
            if (!cand)
                continue;
            const int o = s ^ (rot << 1);
            int32_t u[Cols<RT>::N];
            load_units_stage<RT, F>(sp.units + (size_t)(base + o) * c.R, u, c.R);
            const long long k = order_key(exact_score<RT, G>(u, sp.vals[base + o], 0, c.sp, c.R, c.rg));
            if (k < key || (k == key && loc0 + o < bi)) {
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
        load_units_stage<RT, F>(sp.units + (size_t)i * c.R, uw, c.R);
        take_winner<RT, G>(c, job, bi, uw, sp.vals[i], 0, true, key_value(key));
        atomicAdd(c.st.stats, 1ull);
    }
}

// Tile of a table whose jobs all have K options, K in {4, 8, 16, 32}. Each lane evaluates 4
// consecutive options of one job (a tile row block is 128 options), keeps their smallest and
// second-smallest screen values, and a log2(K / 4)-step xor butterfly over the job's K / 4 lanes
// completes the job. An unambiguous job's winner is the unique option holding the smallest value.
template <int RT, bool G, bool F>
__device__ void process_tile_uniform4(WarpCtx<RT, G> &c, const TileDesc &d, const StagePtrs &sp, int lane)
{
    const int R = c.R;
    const int n = d.n_opt;
    const int K = c.uniform_k;
    const int KL = K >> 2;                  // lanes per job
    for (int b = 0; b < n; b += 128) {
        const int base = b + 4 * lane;
        const bool valid = base < n;        // n is a multiple of K, hence of 4
        const int rot = 0;   // measured slower with the half swap on this path
        float q[4] = {INFINITY, INFINITY, INFINITY, INFINITY};
        uint32_t dupmask = 0;
        if (valid) {
            int32_t u[4][Cols<RT>::N];
            bool dup[4];
            load_units4_smem<RT>(sp.units + (size_t)base * R, u, dup, R, rot);
            const double2 va = reinterpret_cast<const double2 *>(sp.vals + base)[rot];
            const double2 vb = reinterpret_cast<const double2 *>(sp.vals + base)[rot ^ 1];
            const double v[4] = {va.x, va.y, vb.x, vb.y};
#pragma unroll
            for (int o = 0; o < 4; ++o) {
                dupmask |= dup[o] ? (1u << o) : 0u;
                if (!dup[o])
                    q[o] = screen_score_st<RT, G, F>(u[o], v[o], 0, c.sp, R, c.rg);
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
            // an unambiguous job's smallest value is held by one slot only (a tie would make m2 = m1)
            int w = -1;
#pragma unroll
            for (int o = 3; o >= 0; --o)
                if (q[o] == m1)
                    w = o ^ (rot << 1);
            if (w >= 0) {
                const int i = base + w;
                int32_t uw[Cols<RT>::N];
                load_units_stage<RT, F>(sp.units + (size_t)i * R, uw, R);
                take_winner<RT, G>(c, d.job_begin + (i >> c.log2_k), i & (K - 1), uw, sp.vals[i], 0, false, 0.0);
            }
        }
        const bool lamb = valid && amb;
        if (__any_sync(FULL, lamb))
            resolve4_in_row<RT, G, F>(c, sp, lamb, q, dupmask, thr, base, base & (K - 1),
                                   d.job_begin + (base >> c.log2_k), KL, rot);
    }
}

// Exact resolution inside a row of a run: every lane of an ambiguous job screens its 4 options again
// (the same instructions give the same q) and rescores in fp64 its survivors (q <= thr; every option
// but the duplicates in exact mode), in increasing index order, then an xor butterfly over the job's L
// lanes keeps the lexicographic minimum of (s, job-local index), and the lane holding that option
// records it. base: tile-local index of the lane's first option; loc: its job-local index; lamb: the
// lane's job is ambiguous.
template <int RT, bool G, bool F>
__device__ __forceinline__ void resolve_run_row(WarpCtx<RT, G> &c, const StagePtrs &sp, bool lamb, float thr,
                                                int base, int loc, int64_t job, int L)
{
    long long key = 0x7fffffffffffffffLL;
    int bi = kIdxNone;
    if (lamb) {
        for (int o = 0; o < 4; ++o) {
            int32_t u[Cols<RT>::N];
            if (load_units_stage<RT, F>(sp.units + (size_t)(base + o) * c.R, u, c.R))
                continue;
            const double v = sp.vals[base + o];
            if (!c.sp.exact && !(screen_score<RT, G>(u, v, 0, c.sp, c.R, c.rg) <= thr))
                continue;
            const long long k = order_key(exact_score<RT, G>(u, v, 0, c.sp, c.R, c.rg));
            if (k < key) {
                key = k;
                bi = loc + o;
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
    if (lamb && bi >= loc && bi < loc + 4) {
        const int i = base + (bi - loc);
        int32_t uw[Cols<RT>::N];
        load_units_stage<RT, F>(sp.units + (size_t)i * c.R, uw, c.R);
        take_winner<RT, G>(c, job, bi, uw, sp.vals[i], 0, true, key_value(key));
        atomicAdd(c.st.stats, 1ull);
    }
}

// Tile of a run whose jobs all have K = 4m options, m <= 32. A job owns L = 2^ceil(log2 m) lanes;
// lane `sub` of a job screens its options 4 sub .. 4 sub + 3 (16-byte shared loads: the run starts on
// a 4-option boundary) and folds them, in increasing index order, into its smallest value (with its
// index) and second-smallest value; lanes past the job's end idle. A log2(L)-step xor butterfly of
// (smallest, second smallest) completes the job as in the uniform path; an unambiguous job's winner
// is the unique option holding the smallest value, recorded by the lane that holds it.
template <int RT, bool G, bool F>
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
        const int loc = 4 * sub;
        const bool valid = jl < n_job && sub < m;
        const int base = jl * K + loc;
        const int rot = half_swap<RT>(base);   // slot s holds option s ^ (2 rot)
        float m1 = INFINITY, m2 = INFINITY;
        int i1 = kIdxNone;
        if (valid) {
            int32_t u[4][Cols<RT>::N];
            bool dup[4];
            load_units4_smem<RT>(sp.units + (size_t)base * R, u, dup, R, rot);
            const double2 va = reinterpret_cast<const double2 *>(sp.vals + base)[rot];
            const double2 vb = reinterpret_cast<const double2 *>(sp.vals + base)[rot ^ 1];
            const double v[4] = {va.x, va.y, vb.x, vb.y};
            // m1 and m2 do not depend on the order the slots are taken in; i1 matters only when the
            // smallest value is held by one slot (otherwise m2 = m1 and the job is ambiguous)
#pragma unroll
            for (int o = 0; o < 4; ++o) {
                const float q = dup[o] ? INFINITY : screen_score_st<RT, G, F>(u[o], v[o], 0, c.sp, R, c.rg);
                const bool better = q < m1;
                m2 = better ? m1 : fminf(m2, q);
                i1 = better ? loc + (o ^ (rot << 1)) : i1;
                m1 = fminf(m1, q);
            }
        }
        const float lm1 = m1;
        for (int dd = 1; dd < L; dd <<= 1) {
            const float o1 = __shfl_xor_sync(FULL, m1, dd);
            const float o2 = __shfl_xor_sync(FULL, m2, dd);
            m2 = fminf(fminf(m2, o2), fmaxf(m1, o1));
            m1 = fminf(m1, o1);
        }
        const float thr = __fadd_ru(m1, c.sp.e2);
        const bool amb = c.sp.exact || !(m2 > thr);
        const int64_t job = d.job_begin + jl;
        if (valid && !amb && lm1 == m1) {
            const int i = jl * K + i1;
            int32_t uw[Cols<RT>::N];
            load_units_stage<RT, F>(sp.units + (size_t)i * R, uw, R);
            take_winner<RT, G>(c, job, i1, uw, sp.vals[i], 0, false, 0.0);
        }
        const bool lamb = valid && amb;
        if (__any_sync(FULL, lamb))
            resolve_run_row<RT, G, F>(c, sp, lamb, thr, base, loc, job, L);
    }
}

// Tile of a general table (any job sizes). Rows of 32 options are reduced by a segmented scan:
// heads (first options) and ends (last options) of jobs in the row come from the staged job
// offsets; a job continuing from the previous row enters as a carry; rows entirely inside one job
// only fold per lane. A job larger than a tile arrives as consecutive chunk tiles of this warp
// (big_first / big_carry carry its state across them) and is resolved from global memory.
template <int RT, bool G, bool F>
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
            const bool dup = load_units_stage<RT, F>(sp.units + (size_t)i * R, u, R);
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
            load_option<RT, G, F>(c, !big, sp.units, sp.vals, sp.grp, big ? x.idx : x.idx, big ? big_first : 0, uw, vw,
                               gw);
            take_winner<RT, G>(c, job, li, uw, vw, gw, false, 0.0);
        }
        const uint32_t amask = __ballot_sync(FULL, amb);
        if (amask)
            resolve_row<RT, G, F>(c, lane, amask, big, sp.units, sp.vals, sp.grp, jstart, jend, thr, job, big_first);
    }
    if (big) {
        if (priv_dirty)
            carry = combine(carry, allreduce_best(priv));
        big_carry = carry;
    }
}
// needed. Each lane folds the options it owns (lane-strided: conflict-free shared loads) into a
// lane-private state carried across the job's chunks; the job's last chunk reduces the states across
// the warp once and records the winner (exact resolution from global memory when ambiguous).
template <int RT, bool G, bool F>
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
                    q[o] = screen_score_st<RT, G, F>(u, v, g, c.sp, R, c.rg);
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
        const float q = dup ? INFINITY : screen_score_st<RT, G, F>(u, v, g, c.sp, R, c.rg);
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
            // the winner's data: from the stage when it lies in this (last) chunk, else from global
            // memory (the earlier chunks' stages have been refilled)
            int32_t uw[Cols<RT>::N];
            double vw;
            int gw;
            const bool here = x.idx >= chunk_base;
            load_option<RT, G, F>(c, here, sp.units, sp.vals, sp.grp, here ? x.idx - chunk_base : x.idx, big_first, uw,
                               vw, gw);
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
            load_option<RT, G, F>(c, false, sp.units, sp.vals, sp.grp, big_priv.idx, big_first, u, v, g);
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
            load_option<RT, G, F>(c, false, sp.units, sp.vals, sp.grp, bi, big_first, uw, vw, gw);
            take_winner<RT, G>(c, d.job_begin, bi, uw, vw, gw, true, key_value(key));
            atomicAdd(c.st.stats, 1ull);
        }
    } else {
        resolve_row<RT, G, F>(c, lane, 1u, true, sp.units, sp.vals, sp.grp, 0, K, thr, d.job_begin, big_first);
    }
}
}  // namespace

}  // namespace esp
