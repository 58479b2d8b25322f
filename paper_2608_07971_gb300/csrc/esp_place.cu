// Factored placement kernels of the ESP tatonnement (Sec. 3.2 with the placement expansion of
// Sec. 3.3): one pass over configurations x nodes per launch (k_place), and all rounds in one
// cooperative launch (k_place_res).

#include <algorithm>
#include <cmath>
#include <cstdint>
#include <cuda_runtime.h>

#include "esp_device.cuh"
#include "esp_kernels.h"
#include "esp_place.h"
#include "esp_warp.cuh"

namespace esp {

namespace {

// ---------------------------------------------------------------------------------------------
// Factored placement evaluation (esp_load_placement). A job's options are its KC configurations
// crossed with N nodes, and only the configurations are stored (Sec. 3.3's slowdown enters the
// value of (k, n) as the fp32 penalty sens_j * D[a_j][b_n]): a pass reads a few hundred bytes per
// job instead of KC * N options. One warp per job at a time; lane l takes nodes l and l + 32.
//
// Screen. G_k = the fp32 chain over the globally priced columns from -v32_k (v truncated as for a
// stored option), and candidate (k, n) scores q = the fp32 chain over the node's columns from
// fl(G_k + pen_n). Against the exact s (the fp64 chain from -(v_k - (double)pen_n)) this is one
// rounding more than the screen of a stored option; with M_s >= max|v_k| + max pen + sum_r max p_r
// max u_r the error stays within the same E (which has a factor of about 4 to spare), so the
// screen rule and the exact rule are those of the streaming kernel. Candidates are visited in
// increasing local index k * N + n on every lane, and configurations that repeat an earlier one
// of their job (marked at load) are skipped: their twins have lower indices and equal scores.

__host__ __device__ inline int place_warp_bytes(int R, int P, int KC)
{
    // configuration units, values, fp32 global parts, fp32 node-column units, fp32 prices
    return round16(KC * R * 4) + round16(KC * 8) + round16(KC * 4) + round16(KC * R * 4) + round16(P * 4);
}

template <int RT>
__device__ __forceinline__ float place_global_part(const int32_t *u, double v, const ScenarioPrices &sp, int rg)
{
    float g = -screen_value(v);
#pragma unroll
    for (int r = 0; r < Cols<RT>::N; ++r) {
        if (r >= rg)
            break;
        g = __fmaf_rn(sp.pf[r], __int2float_rn(u[r]), g);
    }
    return g;
}

// uf: the configuration's units in fp32 (exact below 2^24, rounded above, as the stored screen does)
template <int RT>
__device__ __forceinline__ float place_node_part(const float *uf, float base, const float *p32s, int rg, int R, int n)
{
    float q = base;
    for (int r = rg; r < R; ++r)
        q = __fmaf_rn(p32s[rg + (R - rg) * n + (r - rg)], uf[r], q);
    return q;
}

// Shared-memory areas of one warp of the placement kernels: configuration units, values, fp32
// global parts, fp32 node-column units, fp32 prices.
struct PlaceWarpSmem {
    int32_t *us;
    double *vs;
    float *gs;
    float *ufs;
    float *p32s;
};

__device__ __forceinline__ PlaceWarpSmem place_warp_smem(unsigned char *smem, int wid, int R, int P, int KC)
{
    unsigned char *wbase = smem + (size_t)wid * place_warp_bytes(R, P, KC);
    PlaceWarpSmem w;
    w.us = reinterpret_cast<int32_t *>(wbase);
    w.vs = reinterpret_cast<double *>(wbase + round16(KC * R * 4));
    w.gs = reinterpret_cast<float *>(wbase + round16(KC * R * 4) + round16(KC * 8));
    w.ufs = reinterpret_cast<float *>(wbase + round16(KC * R * 4) + round16(KC * 8) + round16(KC * 4));
    w.p32s = reinterpret_cast<float *>(wbase + 2 * round16(KC * R * 4) + round16(KC * 8) + round16(KC * 4));
    return w;
}

// Best responses of the jobs [j_begin, j_end) (global job indices) over their configurations x
// nodes at the prices of c, the winners' demand into c's accumulators, then a flush.
template <int RT>
__device__ void place_jobs(WarpCtx<RT, true> &c, const DevPlace &pl, const PlaceWarpSmem &ws, int64_t j_begin,
                           int64_t j_end, int lane)
{
    const DevTable &t = c.t;
    const DevState &st = c.st;
    const int KC = pl.KC, N = pl.N, NT = pl.NT;
    const int R = c.R, rg = c.rg;
    int32_t *us = ws.us;
    double *vs = ws.vs;
    float *gs = ws.gs;
    float *ufs = ws.ufs;
    float *p32s = ws.p32s;
    for (int64_t j = j_begin; j < j_end; ++j) {
        const int sc = (int)(j / t.J);
        if (sc != c.s)
            enter_scenario<RT, true>(c, sc, p32s, lane);
        if (c.sp.skip)
            continue;
        __syncwarp();
        for (int i = lane; i < KC * R; i += 32)
            us[i] = __ldg(pl.cfg_units + j * KC * R + i);
        for (int k = lane; k < KC; k += 32)
            vs[k] = __ldg(pl.cfg_values + j * KC + k);
        const float sens = __ldg(pl.sens + j);
        const int aj = __ldg(pl.job_type + j);
        const uint32_t dup = __ldg(pl.cfg_dup + j);
        __syncwarp();
        // the global part of every configuration once (lane k), and the node columns' units in fp32;
        // a repeated configuration gets +inf and never survives the screen
        for (int k = lane; k < KC; k += 32)
            gs[k] = ((dup >> k) & 1u) ? INFINITY : place_global_part<RT>(us + k * R, vs[k], c.sp, rg);
        for (int i = lane; i < KC * R; i += 32)
            ufs[i] = __int2float_rn(us[i]);
        __syncwarp();

        const int n0 = lane, n1 = lane + 32;
        const bool h0 = n0 < N, h1 = n1 < N;
        const float pen0 = h0 ? __fmul_rn(sens, __ldg(pl.D + aj * NT + __ldg(pl.node_type + n0))) : 0.0f;
        const float pen1 = h1 ? __fmul_rn(sens, __ldg(pl.D + aj * NT + __ldg(pl.node_type + n1))) : 0.0f;
        float m1 = INFINITY, m2 = INFINITY;
        int i1 = kIdxNone;
        auto fold = [&](float q, int idx) {
            const bool better = q < m1;
            m2 = better ? m1 : fminf(m2, q);
            i1 = better ? idx : i1;
            m1 = fminf(m1, q);
        };
        for (int k = 0; k < KC; ++k) {
            const float g = gs[k];
            const float *uk = ufs + k * R;
            if (h0)
                fold(place_node_part<RT>(uk, __fadd_rn(g, pen0), p32s, rg, R, n0), k * N + n0);
            if (h1)
                fold(place_node_part<RT>(uk, __fadd_rn(g, pen1), p32s, rg, R, n1), k * N + n1);
        }
        const Best x = allreduce_best(Best{m1, i1, m2});
        const float thr = __fadd_ru(x.m1, c.sp.e2);
        int win = x.idx;
        double s_w = 0.0;
        bool has_s = false;
        if (c.sp.exact || !(x.m2 > thr)) {
            // survivors rescored in fp64: v_kn = v_k - (double)pen_n, then the chain of Eq. esp_score
            long long key = 0x7fffffffffffffffLL;
            int bi = kIdxNone;
            for (int k = 0; k < KC; ++k) {
                if ((dup >> k) & 1u)
                    continue;
                const int32_t *uk = us + k * R;
                int32_t u[Cols<RT>::N];
#pragma unroll
                for (int r = 0; r < Cols<RT>::N; ++r)
                    u[r] = (RT != 0 || r < R) ? uk[r] : 0;
                const float g = gs[k];
#pragma unroll
                for (int h = 0; h < 2; ++h) {
                    const int n = h ? n1 : n0;
                    if (!(h ? h1 : h0))
                        continue;
                    const float pen = h ? pen1 : pen0;
                    const float q = place_node_part<RT>(ufs + k * R, __fadd_rn(g, pen), p32s, rg, R, n);
                    if (!c.sp.exact && !(q <= thr))
                        continue;
                    const double v = __dsub_rn(vs[k], (double)pen);
                    const long long kk = order_key(exact_score<RT, true>(u, v, n, c.sp, R, rg));
                    if (kk < key) {
                        key = kk;
                        bi = k * N + n;
                    }
                }
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
            win = bi;
            s_w = key_value(key);
            has_s = true;
            if (lane == 0)
                atomicAdd(st.stats, 1ull);
        }
        if (lane == 0) {
            const int k = win / N, n = win - k * N;
            int32_t u[Cols<RT>::N];
#pragma unroll
            for (int r = 0; r < Cols<RT>::N; ++r)
                u[r] = (RT != 0 || r < R) ? us[k * R + r] : 0;
            const double v = __dsub_rn(vs[k], (double)__fmul_rn(sens, __ldg(pl.D + aj * NT + __ldg(pl.node_type + n))));
            take_winner<RT, true>(c, j, win, u, v, n, has_s, s_w);
        }
    }
    flush<RT, true>(c, lane);
}

template <int RT, bool PLAIN>
__global__ void __launch_bounds__(kPlaceWarps * 32, 4) k_place(DevTable t, DevState st, DevPlace pl, SolveArgs a,
                                                            int round, int kind)
{
    extern __shared__ __align__(16) unsigned char smem[];
    const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
    const int R = RT ? RT : t.R, rg = t.r_global;
    const PlaceWarpSmem ws = place_warp_smem(smem, wid, R, t.P, pl.KC);
    const int w = blockIdx.x * kPlaceWarps + wid;
    if (w >= pl.n_warps)
        return;

    WarpCtx<RT, true> c;
    c.persist = false;
    c.scen_tiles = nullptr;
    c.ntiles = 0;
    c.t = t;
    c.st = st;
    c.scen_warps = pl.scen_warps;
    c.a = a;
    c.round = round;
    c.R = R;
    c.rg = rg;
    c.kind = PLAIN ? (int)PASS_ROUND : kind;
    c.want_min = PLAIN ? false : ((kind == PASS_FINAL) || (st.dual_trace != nullptr));
    c.want_hash = PLAIN ? false : ((kind == PASS_ROUND) && (st.hash_trace != nullptr));
    c.uniform_k = 0;
    c.log2_k = 0;
    c.s = -1;
#pragma unroll
    for (int r = 0; r < Cols<RT>::N; ++r)
        c.acc[r] = 0;
    c.hacc = 0;
    place_jobs<RT>(c, pl, ws, pl.warp_job[w], pl.warp_job[w + 1], lane);
}

// Grid-wide barrier of a cooperative launch: every CTA adds 1 to *bar and waits until it reaches
// target (= CTAs x barriers so far). Thread 0 waits, bounded (about 4 s); on expiry, or when
// another CTA gave up (bar[1] != 0), the barrier fails for the whole CTA, the device error word is
// flagged and bar[1] set so that no CTA waits for it any longer.
__device__ bool grid_barrier(unsigned int *bar, unsigned int target, unsigned int *err, int *ok_s)
{
    __threadfence();
    __syncthreads();
    if (threadIdx.x == 0) {
        atomicAdd(bar, 1u);
        uint64_t t0;
        asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t0));
        bool ok = false;
        for (uint32_t it = 0;; ++it) {
            unsigned int v, ab;
            asm volatile("ld.acquire.gpu.u32 %0, [%1];" : "=r"(v) : "l"(bar) : "memory");
            if ((int)(v - target) >= 0) {
                ok = true;
                break;
            }
            asm volatile("ld.relaxed.gpu.u32 %0, [%1];" : "=r"(ab) : "l"(bar + 1) : "memory");
            if (ab != 0u)
                break;
            if (it > 64) {
                uint64_t t1;
                asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t1));
                if (t1 - t0 > 4000000000ull)
                    break;
                __nanosleep(200);
            }
        }
        if (!ok) {
            atomicOr(err, DEV_ERR_TIMEOUT);
            atomicExch(bar + 1, 1u);
        }
        *ok_s = ok ? 1 : 0;
    }
    __syncthreads();
    return *ok_s != 0;
}

// Exact score of Eq. esp_score (the chain of exact_score) with the prices in shared memory.
template <int RT>
__device__ __forceinline__ double exact_score_shared(const int32_t *u, double v, int g, const double *p64, int R,
                                                     int rg)
{
    double s = -v;
#pragma unroll
    for (int r = 0; r < Cols<RT>::N; ++r) {
        if (RT == 0 && r >= R)
            break;
        s = __fma_rn(p64[r >= rg ? rg + (R - rg) * g + (r - rg) : r], __int2double_rn(u[r]), s);
    }
    return s;
}

// All T rounds of a placement solve in one cooperative launch of one CTA (kPlaceResWarps warps)
// per SM. Each warp holds its (at most kPlaceResJobs) jobs in shared memory for the whole solve:
// configuration units (int32 and fp32), values, and per lane the penalties of its two nodes. Each
// CTA holds the whole price state of every scenario in shared memory (S * P <= kPlaceResMaxPrices).
// A round: best responses of the CTA's jobs (the arithmetic of k_place), their demand summed in
// shared memory and added to buffer round % 3 of U3 with one atomic per column, a grid barrier,
// then Eq. price_update by the whole CTA from the same totals (one price per thread; per-scenario
// maxima and flags through shared atomics, which are order-independent), identical in every CTA.
// CTA 0 writes the price and demand trajectories, clears the buffer that was last read before this
// round's barrier, and publishes the final state for the final pass. Hash and dual traces are not
// supported here (the host keeps the per-round launches for them).
template <int RT>
__global__ void __launch_bounds__(kPlaceResWarps * 32, 1) k_place_res(DevTable t, DevState st, DevPlace pl,
                                                                   SolveArgs a, PlaceRes pr)
{
    extern __shared__ __align__(16) unsigned char smem[];
    __shared__ int ok_s;
    const int tid = threadIdx.x, lane = tid & 31, wid = tid >> 5;
    const int R = RT ? RT : t.R, rg = t.r_global;
    const int S = t.S, P = t.P, SP = S * P, T = a.T;
    const int KC = pl.KC, N = pl.N, NT = pl.NT;
    const PlaceResLayout L = place_res_layout(S, P, KC, R);

    unsigned long long *Uc = reinterpret_cast<unsigned long long *>(smem + L.u);
    double *lam_s = reinterpret_cast<double *>(smem + L.lam);
    double *p64_s = reinterpret_cast<double *>(smem + L.p64);
    double *capd_s = reinterpret_cast<double *>(smem + L.capd);
    long long *cap_s = reinterpret_cast<long long *>(smem + L.cap);
    float *p32_s = reinterpret_cast<float *>(smem + L.p32);
    float *eb_s = reinterpret_cast<float *>(smem + L.eb);
    int *frozen_s = reinterpret_cast<int *>(smem + L.flags);
    int *status_s = frozen_s + S, *conv_s = frozen_s + 2 * S, *rounds_s = frozen_s + 3 * S;
    int *bad_s = frozen_s + 4 * S, *huge_s = frozen_s + 5 * S;
    unsigned long long *dmax_s = reinterpret_cast<unsigned long long *>(smem + L.maxes);
    unsigned long long *amax_s = dmax_s + S;
    unsigned char *wb = smem + L.warps + (size_t)wid * L.warp_bytes;
    float *gs = reinterpret_cast<float *>(wb);

    // ---- the price state from k_init, and this warp's jobs
    for (int i = tid; i < SP; i += blockDim.x) {
        lam_s[i] = st.lam[i];
        p64_s[i] = st.p64[i];
        p32_s[i] = st.p32[i];
        cap_s[i] = t.cap[i];
        capd_s[i] = (double)t.cap[i];
        Uc[i] = 0ull;
    }
    for (int i = tid; i < S; i += blockDim.x) {
        eb_s[i] = st.ebound[i];
        frozen_s[i] = st.frozen[i];
        status_s[i] = 0;
        conv_s[i] = 0;
        rounds_s[i] = 0;
        bad_s[i] = 0;
        huge_s[i] = 0;
        dmax_s[i] = 0ull;
        amax_s[i] = 0ull;
    }
    const int w = blockIdx.x * kPlaceResWarps + wid;
    const int64_t j0 = (w < pr.n_warps) ? pr.warp_job[w] : 0;
    const int nj = (w < pr.n_warps) ? (int)(pr.warp_job[w + 1] - j0) : 0;
    const int n0 = lane, n1 = lane + 32;
    const bool h0 = n0 < N, h1 = n1 < N;
    float pen0[kPlaceResJobs], pen1[kPlaceResJobs];
    uint32_t dup[kPlaceResJobs];
    int scen[kPlaceResJobs];
#pragma unroll
    for (int q = 0; q < kPlaceResJobs; ++q) {
        pen0[q] = pen1[q] = 0.0f;
        dup[q] = 0u;
        scen[q] = 0;
        if (q < nj) {
            const int64_t j = j0 + q;
            scen[q] = (int)(j / t.J);
            int32_t *us = reinterpret_cast<int32_t *>(wb + L.job_units + q * L.job_bytes);
            float *ufs = reinterpret_cast<float *>(wb + L.job_ufs + q * L.job_bytes);
            double *vs = reinterpret_cast<double *>(wb + L.job_vals + q * L.job_bytes);
            for (int i = lane; i < KC * R; i += 32) {
                const int32_t u = __ldg(pl.cfg_units + j * KC * R + i);
                us[i] = u;
                ufs[i] = __int2float_rn(u);
            }
            for (int k = lane; k < KC; k += 32)
                vs[k] = __ldg(pl.cfg_values + j * KC + k);
            const float sens = __ldg(pl.sens + j);
            const int aj = __ldg(pl.job_type + j);
            dup[q] = __ldg(pl.cfg_dup + j);
            pen0[q] = h0 ? __fmul_rn(sens, __ldg(pl.D + aj * NT + __ldg(pl.node_type + n0))) : 0.0f;
            pen1[q] = h1 ? __fmul_rn(sens, __ldg(pl.D + aj * NT + __ldg(pl.node_type + n1))) : 0.0f;
            float *pens = reinterpret_cast<float *>(wb + L.job_pens + q * L.job_bytes);
            pens[n0] = pen0[q];
            pens[n1] = pen1[q];
        }
    }
    __syncthreads();

    for (int round = 0; round < T; ++round) {
        unsigned long long *Ub = pr.U3 + (size_t)(round % 3) * SP;

        // ---- best responses of this warp's jobs at the CTA's prices
#pragma unroll
        for (int q = 0; q < kPlaceResJobs; ++q) {
            if (q >= nj)
                break;
            const int sc = scen[q];
            if (frozen_s[sc])
                continue;
            const int32_t *us = reinterpret_cast<const int32_t *>(wb + L.job_units + q * L.job_bytes);
            const float *ufs = reinterpret_cast<const float *>(wb + L.job_ufs + q * L.job_bytes);
            const double *vs = reinterpret_cast<const double *>(wb + L.job_vals + q * L.job_bytes);
            const float *p32s = p32_s + (size_t)sc * P;
            const double *p64s = p64_s + (size_t)sc * P;
            ScenarioPrices sp;
#pragma unroll
            for (int r = 0; r < Cols<RT>::N; ++r)
                sp.pf[r] = (r < rg) ? p32s[r] : 0.0f;
            const float e = eb_s[sc];
            sp.exact = !(e < INFINITY);
            sp.e2 = sp.exact ? INFINITY : 2.0f * e;
            __syncwarp();
            for (int k = lane; k < KC; k += 32)
                gs[k] = ((dup[q] >> k) & 1u) ? INFINITY : place_global_part<RT>(us + k * R, vs[k], sp, rg);
            __syncwarp();
            const float pa = pen0[q], pb = pen1[q];
            const float *pens = reinterpret_cast<const float *>(wb + L.job_pens + q * L.job_bytes);
            // this lane's node prices (columns r >= rg of nodes n0, n1) in registers
            const int nc = R - rg;
            float pn0[Cols<RT>::N], pn1[Cols<RT>::N];
#pragma unroll
            for (int c2 = 0; c2 < Cols<RT>::N; ++c2) {
                pn0[c2] = (c2 < nc && h0) ? p32s[rg + nc * n0 + c2] : 0.0f;
                pn1[c2] = (c2 < nc && h1) ? p32s[rg + nc * n1 + c2] : 0.0f;
            }
            // q of (k, n0) and (k, n1): the chain of place_node_part, same operations in the same order
            auto node_q = [&](int k, float &q0, float &q1) {
                const float g = gs[k];
                const float *uk = ufs + k * R + rg;
                q0 = __fadd_rn(g, pa);
                q1 = __fadd_rn(g, pb);
#pragma unroll
                for (int c2 = 0; c2 < Cols<RT>::N; ++c2) {
                    if (c2 >= nc)
                        break;
                    const float uf = uk[c2];
                    q0 = __fmaf_rn(pn0[c2], uf, q0);
                    q1 = __fmaf_rn(pn1[c2], uf, q1);
                }
            };
            float m1 = INFINITY, m2 = INFINITY;
            int i1 = kIdxNone;
            auto fold = [&](float qv, int idx) {
                const bool better = qv < m1;
                m2 = better ? m1 : fminf(m2, qv);
                i1 = better ? idx : i1;
                m1 = fminf(m1, qv);
            };
#pragma unroll 4
            for (int k = 0; k < KC; ++k) {
                float q0, q1;
                node_q(k, q0, q1);
                if (h0)
                    fold(q0, k * N + n0);
                if (h1)
                    fold(q1, k * N + n1);
            }
            const Best x = allreduce_best(Best{m1, i1, m2});
            const float thr = __fadd_ru(x.m1, sp.e2);
            int win = x.idx;
            if (sp.exact || !(x.m2 > thr)) {
                // survivors (q <= thr; all in exact mode; repeated configurations never), listed in
                // (k, node half, lane) order; up to 32 are rescored in fp64 one per lane
                int *cand = reinterpret_cast<int *>(wb + L.cand);
                int total = 0;
                for (int k = 0; k < KC && total <= 32; ++k) {
                    if ((dup[q] >> k) & 1u)
                        continue;
                    float q0, q1;
                    node_q(k, q0, q1);
                    const unsigned b0 = __ballot_sync(FULL, h0 && (sp.exact || q0 <= thr));
                    const unsigned b1 = __ballot_sync(FULL, h1 && (sp.exact || q1 <= thr));
                    const unsigned below = (1u << lane) - 1u;
                    const int i0 = total + __popc(b0 & below), i1s = total + __popc(b0) + __popc(b1 & below);
                    if (((b0 >> lane) & 1u) && i0 < 32)
                        cand[i0] = k * N + n0;
                    if (((b1 >> lane) & 1u) && i1s < 32)
                        cand[i1s] = k * N + n1;
                    total += __popc(b0) + __popc(b1);
                }
                __syncwarp();
                long long key = 0x7fffffffffffffffLL;
                int bi = kIdxNone;
                if (total <= 32) {
                    if (lane < total) {
                        const int ci = cand[lane];
                        const int k = ci / N, n = ci - k * N;
                        int32_t u[Cols<RT>::N];
#pragma unroll
                        for (int r = 0; r < Cols<RT>::N; ++r)
                            u[r] = (RT != 0 || r < R) ? us[k * R + r] : 0;
                        const double v = __dsub_rn(vs[k], (double)pens[n]);
                        key = order_key(exact_score_shared<RT>(u, v, n, p64s, R, rg));
                        bi = ci;
                    }
                } else {
                    // many survivors: each lane rescores its own
                    for (int k = 0; k < KC; ++k) {
                        if ((dup[q] >> k) & 1u)
                            continue;
                        float q0, q1;
                        node_q(k, q0, q1);
                        const int32_t *uk = us + k * R;
                        int32_t u[Cols<RT>::N];
#pragma unroll
                        for (int r = 0; r < Cols<RT>::N; ++r)
                            u[r] = (RT != 0 || r < R) ? uk[r] : 0;
#pragma unroll
                        for (int h = 0; h < 2; ++h) {
                            const int n = h ? n1 : n0;
                            if (!(h ? h1 : h0))
                                continue;
                            if (!sp.exact && !((h ? q1 : q0) <= thr))
                                continue;
                            const double v = __dsub_rn(vs[k], (double)(h ? pb : pa));
                            const long long kk = order_key(exact_score_shared<RT>(u, v, n, p64s, R, rg));
                            if (kk < key) {
                                key = kk;
                                bi = k * N + n;
                            }
                        }
                    }
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
                __syncwarp();
                win = bi;
                if (lane == 0)
                    atomicAdd(st.stats, 1ull);
            }
            // the winner's units into the CTA's demand (lane r: column r)
            const int kw = win / N, nw = win - kw * N;
            if (lane < R) {
                const long long u = us[kw * R + lane];
                const int col = lane >= rg ? rg + (R - rg) * nw + (lane - rg) : lane;
                if (u != 0)
                    atomicAdd(Uc + (size_t)sc * P + col, (unsigned long long)u);
            }
        }
        __syncthreads();
        // ---- the CTA's demand into the round's buffer; per-scenario reductions reset
        for (int i = tid; i < SP; i += blockDim.x) {
            const unsigned long long v = Uc[i];
            if (v != 0ull) {
                atomicAdd(Ub + i, v);
                Uc[i] = 0ull;
            }
        }
        for (int i = tid; i < S; i += blockDim.x) {
            bad_s[i] = 0;
            huge_s[i] = 0;
            dmax_s[i] = 0ull;
            amax_s[i] = 0ull;
        }
        if (!grid_barrier(pr.bar, (unsigned int)(round + 1) * gridDim.x, st.err, &ok_s))
            break;

        // ---- Eq. price_update of every scenario, one price per thread: the new prices are computed
        // into registers, and written once no price of the scenario became non-finite
        const double eta = step_size(a.eta0, a.step, round);
        const bool lead = blockIdx.x == 0;
        double nl_r[kPlaceResPricesPerThread], pe_r[kPlaceResPricesPerThread];
#pragma unroll
        for (int m = 0; m < kPlaceResPricesPerThread; ++m) {
            const int i = tid + m * kPlaceResWarps * 32;
            nl_r[m] = pe_r[m] = 0.0;
            if (i >= SP)
                break;
            const int sc = i / P;
            if (frozen_s[sc])
                continue;
            const long long U = (long long)__ldcg(Ub + i);
            if (lead && st.dem_trace)
                st.dem_trace[((size_t)sc * T + round) * P + (i - sc * P)] = U;
            const double lam = lam_s[i];
            const double nl = price_step(lam, U, cap_s[i], capd_s[i], eta, a.mode);
            nl_r[m] = nl;
            pe_r[m] = effective_price(nl, capd_s[i], a.mode);
            if (!isfinite(nl))
                atomicOr(bad_s + sc, 1);
            if (a.tol > 0.0) {   // maxima of the stopping rule (non-negative doubles order as integers)
                atomicMax(dmax_s + sc, (unsigned long long)__double_as_longlong(fabs(nl - lam)));
                atomicMax(amax_s + sc, (unsigned long long)__double_as_longlong(fabs(lam)));
            }
        }
        __syncthreads();
#pragma unroll
        for (int m = 0; m < kPlaceResPricesPerThread; ++m) {
            const int i = tid + m * kPlaceResWarps * 32;
            if (i >= SP)
                break;
            const int sc = i / P;
            if (frozen_s[sc] || bad_s[sc])
                continue;
            lam_s[i] = nl_r[m];
            if (lead && st.lam_trace)
                st.lam_trace[((size_t)sc * (T + 1) + round + 1) * P + (i - sc * P)] = nl_r[m];
            p64_s[i] = pe_r[m];
            p32_s[i] = __double2float_rn(pe_r[m]);
            if (!(pe_r[m] <= 0x1p100))
                atomicOr(huge_s + sc, 1);
        }
        __syncthreads();
        // stopping rule and screen bound, one warp per scenario (the summation order of set_prices)
        for (int sc = wid; sc < S; sc += kPlaceResWarps) {
            if (frozen_s[sc])
                continue;
            if (bad_s[sc]) {
                if (lane == 0) {
                    status_s[sc] = 2;
                    frozen_s[sc] = 1;
                }
                continue;
            }
            const double dmax = __longlong_as_double((long long)dmax_s[sc]);
            const double amax = __longlong_as_double((long long)amax_s[sc]);
            const bool conv = (a.tol > 0.0) && (dmax <= a.tol * fmax(1.0, amax));
            const double *p64s = p64_s + (size_t)sc * P;
            double term = 0.0;
            const int rgm = (t.n_groups == 0) ? R : rg;
            if (lane < rgm)
                term = p64s[lane] * (double)st.umax[(size_t)sc * R + lane];
            for (int c2 = 0; c2 < R - rgm; ++c2) {
                double pm = 0.0;
                for (int gi = lane; gi < t.n_groups; gi += 32)
                    pm = fmax(pm, p64s[rgm + (R - rgm) * gi + c2]);
                pm = warp_max(pm);
                if (lane == rgm + c2)
                    term = pm * (double)st.umax[(size_t)sc * R + lane];
            }
            const double M = st.vmax[sc] + warp_sum_fixed(term);
            if (lane == 0) {
                if (lead && st.time_trace)
                    st.time_trace[(size_t)sc * T + round] = global_ns();
                rounds_s[sc] = round + 1;
                if (conv) {
                    conv_s[sc] = 1;
                    frozen_s[sc] = 1;
                }
                eb_s[sc] = screen_bound(M, R, a.exact_only || huge_s[sc] != 0);
            }
        }
        if (lead) {   // buffer (round + 2) % 3 was last read before this round's barrier
            unsigned long long *Uz = pr.U3 + (size_t)((round + 2) % 3) * SP;
            for (int i = tid; i < SP; i += blockDim.x)
                Uz[i] = 0ull;
        }
        __syncthreads();
    }
    // ---- CTA 0 publishes the final price state for the final pass and the objectives
    if (blockIdx.x == 0) {
        for (int i = tid; i < SP; i += blockDim.x) {
            st.lam[i] = lam_s[i];
            st.p64[i] = p64_s[i];
            st.p32[i] = p32_s[i];
        }
        for (int i = tid; i < S; i += blockDim.x) {
            st.ebound[i] = eb_s[i];
            st.frozen[i] = frozen_s[i];
            st.status[i] = status_s[i];
            st.converged[i] = conv_s[i];
            st.rounds_run[i] = rounds_s[i];
        }
    }
}

}  // namespace

int place_smem_bytes(int R, int P, int KC, int N, int NT)
{
    (void)N;
    (void)NT;
    return kPlaceWarps * place_warp_bytes(R, P, KC);
}

template <typename F>
static auto place_dispatch(int R, bool plain, F &&f)
{
    if (R == 8)
        return plain ? f(reinterpret_cast<const void *>(&k_place<8, true>)) : f(reinterpret_cast<const void *>(&k_place<8, false>));
    return plain ? f(reinterpret_cast<const void *>(&k_place<0, true>)) : f(reinterpret_cast<const void *>(&k_place<0, false>));
}

int place_ctas_per_sm(int R, int P, int KC, int N, int NT)
{
    const int smem = place_smem_bytes(R, P, KC, N, NT);
    int best = 1 << 30;
    for (int plain = 0; plain < 2; ++plain) {
        const int n = place_dispatch(R, plain != 0, [&](const void *fn) -> int {
            if (cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, smem) != cudaSuccess)
                return 0;
            int m = 0;
            if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&m, fn, kPlaceWarps * 32, smem) != cudaSuccess)
                return 0;
            return m;
        });
        best = n < best ? n : best;
    }
    return best;
}

cudaError_t launch_place(const DevTable &t, const DevState &st, const DevPlace &pl, const SolveArgs &a, int round,
                         PassKind kind, int grid, cudaStream_t stream)
{
    const int smem = place_smem_bytes(t.R, t.P, pl.KC, pl.N, pl.NT);
    const bool plain = kind == PASS_ROUND && st.hash_trace == nullptr && st.dual_trace == nullptr;
    if (t.R == 8) {
        if (plain)
            k_place<8, true><<<grid, kPlaceWarps * 32, smem, stream>>>(t, st, pl, a, round, kind);
        else
            k_place<8, false><<<grid, kPlaceWarps * 32, smem, stream>>>(t, st, pl, a, round, kind);
    } else {
        if (plain)
            k_place<0, true><<<grid, kPlaceWarps * 32, smem, stream>>>(t, st, pl, a, round, kind);
        else
            k_place<0, false><<<grid, kPlaceWarps * 32, smem, stream>>>(t, st, pl, a, round, kind);
    }
    return cudaGetLastError();
}

int place_res_smem_bytes(int S, int P, int KC, int R)
{
    return place_res_layout(S, P, KC, R).total;
}

int place_res_ctas_per_sm(int S, int P, int KC, int R)
{
    const int smem = place_res_smem_bytes(S, P, KC, R);
    const void *fn = R == 8 ? reinterpret_cast<const void *>(&k_place_res<8>)
                            : reinterpret_cast<const void *>(&k_place_res<0>);
    int m = 0;
    if (cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, smem) != cudaSuccess ||
        cudaOccupancyMaxActiveBlocksPerMultiprocessor(&m, fn, kPlaceResWarps * 32, smem) != cudaSuccess) {
        cudaGetLastError();
        return 0;
    }
    return m;
}

static cudaError_t place_res_launch(const DevTable &t, const DevState &st, const DevPlace &pl, const SolveArgs &a,
                                    const PlaceRes &pr, cudaStream_t stream, bool hold_barrier)
{
    cudaError_t e = cudaMemsetAsync(pr.bar, 0, 2 * sizeof(unsigned int), stream);
    if (e == cudaSuccess && hold_barrier)   // every byte 0xC0: the counter far short of its targets
        e = cudaMemsetAsync(pr.bar, 0xC0, sizeof(unsigned int), stream);
    if (e == cudaSuccess)   // the last rounds of the previous solve leave demand in two buffers
        e = cudaMemsetAsync(pr.U3, 0, 3 * (size_t)t.S * t.P * sizeof(unsigned long long), stream);
    if (e != cudaSuccess)
        return e;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)pr.grid);
    cfg.blockDim = dim3(kPlaceResWarps * 32);
    cfg.dynamicSmemBytes = (size_t)place_res_smem_bytes(t.S, t.P, pl.KC, t.R);
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeCooperative;   // every CTA co-resident: the grid barrier can complete
    attr[0].val.cooperative = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    if (t.R == 8)
        return cudaLaunchKernelEx(&cfg, k_place_res<8>, t, st, pl, a, pr);
    return cudaLaunchKernelEx(&cfg, k_place_res<0>, t, st, pl, a, pr);
}

cudaError_t launch_place_res(const DevTable &t, const DevState &st, const DevPlace &pl, const SolveArgs &a,
                             const PlaceRes &pr, cudaStream_t stream)
{
    return place_res_launch(t, st, pl, a, pr, stream, false);
}

cudaError_t launch_place_res_held(const DevTable &t, const DevState &st, const DevPlace &pl, const SolveArgs &a,
                                  const PlaceRes &pr, cudaStream_t stream)
{
    return place_res_launch(t, st, pl, a, pr, stream, true);
}

}  // namespace esp
