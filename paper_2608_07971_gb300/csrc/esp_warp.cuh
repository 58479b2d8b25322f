// Per-warp evaluation machinery shared by the evaluation-pass kernels (esp_kernels.cu) and the
// factored placement kernels (esp_place.cu) of the ESP tatonnement (Sec. 3.2): the fp32 screen and
// fp64 exact chains of Eq. esp_score, the price update of Eq. price_update with the effective prices
// and screen bound of the next round, a warp's running demand and its flush (with the fused update
// by the last warp of a scenario), and the (m1, index, m2) reduction of the screen.
#pragma once

#include <cmath>
#include <cstdint>
#include <cuda_runtime.h>

#include "esp_device.cuh"
#include "esp_kernels.h"
#include "esp_ptx.cuh"

namespace esp {

namespace {

// ---------------------------------------------------------------------------------------------
// Scoring. Both chains run r = 0 .. R-1 with one correctly rounded fused multiply-add per column.

template <int RT>
struct Cols {
    static constexpr int N = RT ? RT : kMaxR;
};

struct ScenarioPrices {
    float pf[kMaxR];       // fp32 per-unit price of each globally priced stored column
    const float *p32s;     // fp32 prices of the scenario in shared memory (grouped tables)
    const double *p64g;    // fp64 prices of the scenario in global memory
    float e2;              // 2E, +inf: exact evaluation
    bool exact;
    bool skip;             // scenario already stopped
    bool small_units;      // every unit of the table is below 2^23
};

template <int RT, bool G>
__device__ __forceinline__ float screen_score(const int32_t *u, double v, int g, const ScenarioPrices &sp, int R,
                                              int rg)
{
    float q = -screen_value(v);
#pragma unroll
    for (int r = 0; r < Cols<RT>::N; ++r) {
        if (RT == 0 && r >= R)
            break;
        const float price = (G && r >= rg) ? sp.p32s[rg + (R - rg) * g + (r - rg)] : sp.pf[r];
        const float uf = (r < ESP_I2F_COLS) ? __int2float_rn(u[r]) : f32_of_units(u[r], sp.small_units);
        q = __fmaf_rn(price, uf, q);
    }
    return q;
}

template <int RT, bool G>
__device__ __forceinline__ double exact_score(const int32_t *u, double v, int g, const ScenarioPrices &sp, int R,
                                              int rg)
{
    double s = -v;
#pragma unroll
    for (int r = 0; r < Cols<RT>::N; ++r) {
        if (RT == 0 && r >= R)
            break;
        // through L2: a persistent pass sees the prices change between rounds
        const double price = __ldcg(sp.p64g + ((G && r >= rg) ? rg + (R - rg) * g + (r - rg) : r));
        s = __fma_rn(price, __int2double_rn(u[r]), s);
    }
    return s;
}

// Units of one option. The sign bit of column 0 marks an exact duplicate of an earlier option of
// the same job (set at load time; units themselves are >= 0): it is removed here and returned.
template <int RT>
__device__ __forceinline__ bool load_units_smem(const int32_t *p, int32_t *u, int R)
{
    if (RT == 4) {
        const int4 a = *reinterpret_cast<const int4 *>(p);
        u[0] = a.x; u[1] = a.y; u[2] = a.z; u[3] = a.w;
    } else if (RT == 6) {
        const int2 a = reinterpret_cast<const int2 *>(p)[0];
        const int2 b = reinterpret_cast<const int2 *>(p)[1];
        const int2 c = reinterpret_cast<const int2 *>(p)[2];
        u[0] = a.x; u[1] = a.y; u[2] = b.x; u[3] = b.y; u[4] = c.x; u[5] = c.y;
    } else if (RT == 8) {
        const int4 a = reinterpret_cast<const int4 *>(p)[0];
        const int4 b = reinterpret_cast<const int4 *>(p)[1];
        u[0] = a.x; u[1] = a.y; u[2] = a.z; u[3] = a.w; u[4] = b.x; u[5] = b.y; u[6] = b.z; u[7] = b.w;
    } else {
#pragma unroll
        for (int r = 0; r < Cols<RT>::N; ++r)
            u[r] = (r < R) ? p[r] : 0;
    }
    const bool dup = u[0] < 0;
    u[0] &= 0x7fffffff;
    return dup;
}

// Units staged as fp32 bit patterns (F: the tile-interleaved copy of a table whose units are all
// below 2^23, each converted exactly at load; the duplicate mark stays the sign bit of column 0). The
// screen takes them as they are: the same fp32 values the conversion of the integers gives, so the
// same q, without a conversion per unit. Every other use converts them back to the integers.
template <int RT, bool G, bool F>
__device__ __forceinline__ float screen_score_st(const int32_t *u, double v, int g, const ScenarioPrices &sp, int R,
                                                 int rg)
{
    if constexpr (F) {
        static_assert(!G, "fp32 stage units only for tables without a group column");
        float q = -screen_value(v);
#pragma unroll
        for (int r = 0; r < Cols<RT>::N; ++r) {
            if (RT == 0 && r >= R)
                break;
            q = __fmaf_rn(sp.pf[r], __int_as_float(u[r]), q);
        }
        return q;
    } else {
        return screen_score<RT, G>(u, v, g, sp, R, rg);
    }
}

template <int RT, bool F>
__device__ __forceinline__ void stage_units_to_int(int32_t *u, int R)
{
    if constexpr (F) {
#pragma unroll
        for (int r = 0; r < Cols<RT>::N; ++r)
            if (RT != 0 || r < R)
                u[r] = __float2int_rn(__int_as_float(u[r]));
    }
}

// Units of one staged option as integers (duplicate mark removed and returned).
template <int RT, bool F>
__device__ __forceinline__ bool load_units_stage(const int32_t *p, int32_t *u, int R)
{
    const bool dup = load_units_smem<RT>(p, u, R);
    stage_units_to_int<RT, F>(u, R);
    return dup;
}

template <int RT>
__device__ __forceinline__ bool load_units_global(const int32_t *p, int32_t *u, int R)
{
#pragma unroll
    for (int r = 0; r < Cols<RT>::N; ++r)
        u[r] = (RT != 0 || r < R) ? __ldg(p + r) : 0;
    const bool dup = u[0] < 0;
    u[0] &= 0x7fffffff;
    return dup;
}

// ---------------------------------------------------------------------------------------------
// Price update (Eq. price_update), one warp per scenario, and the screen bound of the new prices.

// Effective prices p = lambda (RAW) or lambda / C (NORMALIZED), their fp32 copy, and the bound E.
// A lane's first KEEP prices are unrolled so that their loads and divides overlap (KEEP = 1 where a
// table has at most 32 prices, keeping the evaluation kernels' register budget).
template <int KEEP>
__device__ void set_prices(const DevTable &t, const DevState &st, const SolveArgs &a, int s, int lane)
{
    const int P = t.P, R = t.R;
    bool huge = false;
    auto price_of = [&](int k) {
        const double lam = __ldcg(st.lam + (size_t)s * P + k);
        const double p = effective_price(lam, (double)t.cap[(size_t)s * P + k], a.mode);
        st.p64[(size_t)s * P + k] = p;
        st.p32[(size_t)s * P + k] = __double2float_rn(p);
        huge |= !(p <= 0x1p100);
    };
#pragma unroll
    for (int i = 0; i < KEEP; ++i)
        if (lane + 32 * i < P)
            price_of(lane + 32 * i);
    for (int k = lane + 32 * KEEP; k < P; k += 32)
        price_of(k);
    __syncwarp();
    // M_s = max|v| + sum_r (max price of column r over groups) * (max unit of column r); lane r
    // holds column r's term. The maxima over groups are taken lane-parallel (a max is exact, so the
    // order does not matter).
    double term = 0.0;
    const int rg = (t.n_groups == 0) ? R : t.r_global;
    if (lane < rg)
        term = __ldcg(st.p64 + (size_t)s * P + lane) * (double)st.umax[(size_t)s * R + lane];
    for (int c2 = 0; c2 < R - rg; ++c2) {
        double pm = 0.0;
        for (int gi = lane; gi < t.n_groups; gi += 32)
            pm = fmax(pm, __ldcg(st.p64 + (size_t)s * P + rg + (R - rg) * gi + c2));
        pm = warp_max(pm);
        if (lane == rg + c2)
            term = pm * (double)st.umax[(size_t)s * R + lane];
    }
    const double M = st.vmax[s] + warp_sum_fixed(term);
    huge = __any_sync(FULL, huge);
    if (lane == 0)
        st.ebound[s] = screen_bound(M, R, a.exact_only || huge);
}


// Eq. price_update for scenario s after round `round` (one warp): traces, the projected step, the
// stopping rule, and the prices and screen bound of the next round. Reads what other warps of the
// same launch wrote (demand, minimal reduced costs, fingerprint) through L2. A lane's first KEEP
// new prices are computed once, unrolled (their loads and divides overlap), and kept in registers
// for the write; the rest are recomputed.
// ZERO_U = false leaves the demand in place (a grid-resident solve reads it from every CTA and
// clears it later).
template <int KEEP, bool ZERO_U = true>
__device__ void update_scenario(const DevTable &t, const DevState &st, const SolveArgs &a, int s, int round,
                                int lane)
{
    const int P = t.P, J = t.J, T = a.T;
    const size_t sp = (size_t)s * P;

    if (st.dual_trace) {   // g(lambda^t) from the minimal reduced costs of round t
        double part = 0.0;
        for (int j = lane; j < J; j += 32)
            part += -__ldcg(st.job_min + (size_t)s * J + j);
        double lc = 0.0;
        for (int k = lane; k < P; k += 32)
            lc += (a.mode == 1) ? st.lam[sp + k] : st.lam[sp + k] * (double)t.cap[sp + k];
        const double g = warp_sum_fixed(part) + warp_sum_fixed(lc);
        if (lane == 0) {
            st.dual_trace[(size_t)s * (T + 1) + round] = g;
            if (g < st.best_dual[s])
                st.best_dual[s] = g;
        }
    }
    if (st.hash_trace && lane == 0) {
        st.hash_trace[(size_t)s * T + round] = __ldcg(st.hash + s);
        st.hash[s] = 0ull;
    }

    const double eta = step_size(a.eta0, a.step, round);
    bool bad = false;
    double dmax = 0.0, amax = 0.0;
    double keep[KEEP];
    auto step_of = [&](int k, double &lam_out) {
        const long long U = (long long)__ldcg(st.U + sp + k);
        const long long C = t.cap[sp + k];
        if (st.dem_trace)
            st.dem_trace[((size_t)s * T + round) * P + k] = U;
        lam_out = __ldcg(st.lam + sp + k);
        return price_step(lam_out, U, C, (double)C, eta, a.mode);
    };
#pragma unroll
    for (int i = 0; i < KEEP; ++i) {
        const int k = lane + 32 * i;
        keep[i] = 0.0;
        if (k < P) {
            double lam;
            const double nl = step_of(k, lam);
            keep[i] = nl;
            bad |= !isfinite(nl);
            dmax = fmax(dmax, fabs(nl - lam));
            amax = fmax(amax, fabs(lam));
        }
    }
    for (int k = lane + 32 * KEEP; k < P; k += 32) {
        double lam;
        const double nl = step_of(k, lam);
        bad |= !isfinite(nl);
        dmax = fmax(dmax, fabs(nl - lam));
        amax = fmax(amax, fabs(lam));
    }
    bad = __any_sync(FULL, bad);
    dmax = warp_max(dmax);
    amax = warp_max(amax);
    if (bad) {
        if (ZERO_U)
            for (int k = lane; k < P; k += 32)
                st.U[sp + k] = 0ull;
        if (lane == 0) {
            st.status[s] = 2;
            st.frozen[s] = 1;
        }
        return;
    }
    for (int k = lane, i = 0; k < P; k += 32, ++i) {
        double nl;
        if (i < KEEP) {
#pragma unroll
            for (int q = 0; q < KEEP; ++q)
                if (q == i)
                    nl = keep[q];
        } else {
            const long long U = (long long)__ldcg(st.U + sp + k);
            const long long C = t.cap[sp + k];
            nl = price_step(__ldcg(st.lam + sp + k), U, C, (double)C, eta, a.mode);
        }
        st.lam[sp + k] = nl;
        if (ZERO_U)
            st.U[sp + k] = 0ull;
        if (st.lam_trace)
            st.lam_trace[((size_t)s * (T + 1) + round + 1) * P + k] = nl;
    }
    const bool conv = (a.tol > 0.0) && (dmax <= a.tol * fmax(1.0, amax));
    if (lane == 0) {
        if (st.time_trace)
            st.time_trace[(size_t)s * T + round] = global_ns();
        st.rounds_run[s] = round + 1;
        if (conv) {
            st.converged[s] = 1;
            st.frozen[s] = 1;
        }
    }
    __syncwarp();
    set_prices<KEEP>(t, st, a, s, lane);
}



// ---------------------------------------------------------------------------------------------
// The warp's evaluation context.

template <int RT, bool G>
struct WarpCtx {
    DevTable t;
    DevState st;
    const int32_t *scen_warps;  // non-null: the last warp to finish a scenario in a round pass updates its prices
    SolveArgs a;
    int round;
    int R, rg;
    int kind;                 // PassKind
    bool want_min;            // job_min needed (final pass or dual trace)
    bool want_hash;           // selection fingerprint needed
    int uniform_k;            // > 0: every job has this many options (a power of two <= 32)
    int log2_k;
    int s;                    // current scenario
    bool persist;             // persistent pass: the update publishes the scenario's price version
    const int32_t *scen_tiles;  // persistent pass: tiles of each scenario (arrivals count tiles)
    int ntiles;               // persistent pass: tiles of the current scenario evaluated since the last flush
    ScenarioPrices sp;
    long long acc[Cols<RT>::N];   // per-lane demand of the globally priced columns
    unsigned long long hacc;
};

template <int RT, bool G>
__device__ void flush(WarpCtx<RT, G> &c, int lane)
{
    if (c.s < 0)
        return;
    const int ncol = G ? c.rg : c.R;
    unsigned long long *dst = (c.kind == PASS_ROUND ? c.st.U : c.st.U_final) + (size_t)c.s * c.t.P;
#pragma unroll
    for (int r = 0; r < Cols<RT>::N; ++r) {
        if (r >= ncol)
            break;
        long long v = c.acc[r];
#pragma unroll
        for (int d = 16; d >= 1; d >>= 1)
            v += __shfl_xor_sync(FULL, v, d);
        if (lane == 0 && v != 0)
            atomicAdd(dst + r, (unsigned long long)v);
        c.acc[r] = 0;
    }
    if (c.want_hash) {
        unsigned long long h = c.hacc;
#pragma unroll
        for (int d = 16; d >= 1; d >>= 1)
            h += __shfl_xor_sync(FULL, h, d);
        if (lane == 0)
            atomicAdd(c.st.hash + c.s, h);
        c.hacc = 0;
    }
    if (c.kind == PASS_ROUND && c.scen_warps != nullptr && !c.sp.skip) {
        // arrive; the warp that completes the scenario's count applies Eq. price_update to it. Lane 0
        // issued this warp's demand and fingerprint atomics, so its release-ordered arrival publishes
        // them; with the dual traced, every lane's minimal reduced costs are fenced first.
        if (c.want_min) {
            __syncwarp();
            __threadfence();
        }
        // the persistent pass counts tiles (a warp flushes when its scenario or round changes, whatever
        // the plan's ranges); the round pass counts the plan's warps
        const unsigned int add = c.persist ? (unsigned int)c.ntiles : 1u;
        const unsigned int need = (unsigned int)__ldg((c.persist ? c.scen_tiles : c.scen_warps) + c.s);
        c.ntiles = 0;
        unsigned int old = 0;
        if (lane == 0)
            asm volatile("atom.add.release.gpu.u32 %0, [%1], %2;" : "=r"(old) : "l"(c.st.arrive + c.s), "r"(add)
                         : "memory");
        old = __shfl_sync(FULL, old, 0);
        if (old + add == need) {
            asm volatile("fence.acq_rel.gpu;" ::: "memory");
            update_scenario<G ? 8 : 1>(c.t, c.st, c.a, c.s, c.round, lane);
            if (lane == 0)
                c.st.arrive[c.s] = 0u;     // every warp of this pass has arrived
            if (c.persist) {
                // publish the scenario's next round: every lane's writes (prices, bound, cleared
                // demand) are fenced before lane 0's release of the version; a stopped scenario
                // releases every later round at once (its warps then skip it)
                __threadfence();
                __syncwarp();
                if (lane == 0) {
                    const unsigned int v = c.st.frozen[c.s] ? kVerStopped : (unsigned int)(c.round + 1);
                    asm volatile("st.release.gpu.u32 [%0], %1;" ::"l"(c.st.ver + c.s), "r"(v) : "memory");
                }
            }
        }
    }
}

template <int RT, bool G>
__device__ void enter_scenario(WarpCtx<RT, G> &c, int s, float *p32s_smem, int lane)
{
    flush(c, lane);
    c.s = s;
    const int P = c.t.P;
    c.sp.skip = (c.kind == PASS_ROUND) && (__ldcg(c.st.frozen + s) != 0);
    const float e = __ldcg(c.st.ebound + s);
    c.sp.exact = !(e < INFINITY);
    c.sp.e2 = c.sp.exact ? INFINITY : 2.0f * e;
    c.sp.p64g = c.st.p64 + (size_t)s * P;
    c.sp.small_units = c.t.small_units != 0;
    const int ncol = G ? c.rg : c.R;
#pragma unroll
    for (int r = 0; r < Cols<RT>::N; ++r) {
        const bool have = r < ncol;
        c.sp.pf[r] = have ? __ldcg(c.st.p32 + (size_t)s * P + r) : 0.0f;
    }
    if (G) {
        __syncwarp();
        for (int k = lane; k < P; k += 32)
            p32s_smem[k] = __ldcg(c.st.p32 + (size_t)s * P + k);
        __syncwarp();
        c.sp.p32s = p32s_smem;
    } else {
        c.sp.p32s = nullptr;
    }
}

// The per-job outputs of a winner beyond its demand: fingerprint, final-pass selection and value,
// and its exact reduced cost (computed here unless s64 is given).
template <int RT, bool G>
__device__ __forceinline__ void take_winner_extras(WarpCtx<RT, G> &c, int64_t job, int local, const int32_t *u,
                                                   double v, int g, bool have_s64 = false, double s64 = 0.0)
{
    if (c.t.jmap != nullptr && (c.want_hash || c.want_min || c.kind == PASS_FINAL))
        job = __ldg(c.t.jmap + job);     // sorted layout: outputs go to the caller's job order
    if (c.want_hash)
        c.hacc += splitmix64_mix(((uint64_t)(uint32_t)(job - (int64_t)c.s * c.t.J) << 32) | (uint32_t)local);
    if (c.kind == PASS_FINAL) {
        c.st.sel[job] = local;
        c.st.job_val[job] = v;
    }
    if (c.want_min) {
        if (!have_s64)
            s64 = exact_score<RT, G>(u, v, g, c.sp, c.R, c.rg);
        c.st.job_min[job] = s64;
    }
}

// Records the winner of a job: its demand (per-lane int64 sums; grouped columns straight to the
// scenario's accumulator) and the outputs of take_winner_extras. u/v/g are the winner's data.
template <int RT, bool G>
__device__ __forceinline__ void take_winner(WarpCtx<RT, G> &c, int64_t job, int local, const int32_t *u, double v,
                                            int g, bool have_s64, double s64)
{
    const int R = c.R;
#pragma unroll
    for (int r = 0; r < Cols<RT>::N; ++r) {
        if (RT == 0 && r >= R)
            break;
        if (G && r >= c.rg) {
            unsigned long long *dst = (c.kind == PASS_ROUND ? c.st.U : c.st.U_final) + (size_t)c.s * c.t.P;
            atomicAdd(dst + c.rg + (R - c.rg) * g + (r - c.rg), (unsigned long long)(long long)u[r]);
        } else {
            c.acc[r] += u[r];
        }
    }
    take_winner_extras<RT, G>(c, job, local, u, v, g, have_s64, s64);
}

// Per-job running state of the general (CSR) path: smallest screen value with its index, and the
// smallest value of every other option. Commutative and associative (ties keep the lower index).
struct Best {
    float m1;
    int idx;
    float m2;
};

__device__ __forceinline__ Best best_none() { return Best{INFINITY, kIdxNone, INFINITY}; }

__device__ __forceinline__ Best combine(const Best &a, const Best &b)
{
    const bool take_b = (b.m1 < a.m1) || (b.m1 == a.m1 && b.idx < a.idx);
    return Best{take_b ? b.m1 : a.m1, take_b ? b.idx : a.idx, fminf(fminf(a.m2, b.m2), fmaxf(a.m1, b.m1))};
}

__device__ __forceinline__ Best shfl_up_best(const Best &x, int d)
{
    return Best{__shfl_up_sync(FULL, x.m1, d), __shfl_up_sync(FULL, x.idx, d), __shfl_up_sync(FULL, x.m2, d)};
}

__device__ __forceinline__ Best shfl_best(const Best &x, int src)
{
    return Best{__shfl_sync(FULL, x.m1, src), __shfl_sync(FULL, x.idx, src), __shfl_sync(FULL, x.m2, src)};
}

__device__ __forceinline__ Best allreduce_best(Best x)
{
#pragma unroll
    for (int d = 16; d >= 1; d >>= 1)
        x = combine(x, Best{__shfl_xor_sync(FULL, x.m1, d), __shfl_xor_sync(FULL, x.idx, d),
                            __shfl_xor_sync(FULL, x.m2, d)});
    return x;
}

}  // namespace

}  // namespace esp
