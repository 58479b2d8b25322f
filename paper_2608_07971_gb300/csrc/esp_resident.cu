// Cluster-resident ESP tatonnement (Sec. 3.2.3 of the paper, Alg. 1): every round of a scenario in
// one launch, with the scenario's table held in shared memory.
//
// One thread-block cluster per scenario. Each CTA of the cluster copies a contiguous slice of the
// scenario's jobs (about 1/cs of its options) into its shared memory once and keeps it there for all
// rounds, so a round reads no table bytes from HBM. A round:
//   1. every lane takes whole jobs and scores their options with the fp32 screen; a job whose screen
//      is ambiguous is resolved in fp64 on the same lane (the rule and its proof are those of the
//      streaming kernel: survivors are the options with q <= m1 + 2E, the winner is the lexicographic
//      minimum of (s, index));
//   2. the int64 demands of the winners are summed per warp, then per CTA in warp order;
//   3. each CTA writes its partial into every CTA of the cluster (distributed shared memory) and the
//      cluster meets at one barrier;
//   4. every CTA sums the partials in rank order and applies Eq. price_update itself. The inputs and
//      instructions are the same in every CTA, so all of them hold identical prices without a second
//      exchange; the arithmetic is the streaming path's (esp_device.cuh), so the prices are too.
// After the last round (or the stopping rule) the final evaluation at lambda^T writes the selection,
// the chosen values and the minimal reduced costs, and adds the final demand to U_final.
//
// Partials of round g go to buffer g & 1. A CTA writes buffer g & 1 of its peers only after the
// barrier of round g - 1, which every peer reaches only after it has read buffer (g - 2) & 1, so
// two buffers suffice. No CTA leaves before a last cluster barrier, so no peer writes into the
// shared memory of a finished CTA.

#include <cmath>
#include <cstdint>
#include <cuda_runtime.h>

#include "esp_device.cuh"
#include "esp_kernels.h"
#include "esp_ptx.cuh"

namespace esp {

namespace {

constexpr int kResThreads = kResWarps * 32;
constexpr int kColHash = kMaxR;       // fingerprint word of a partial
constexpr int kColDual = kMaxR + 1;   // dual-sum word of a partial (fp64 bits)

template <int RT>
struct ResCols {
    static constexpr int N = RT ? RT : kMaxR;
};

__device__ __forceinline__ uint32_t cluster_rank()
{
    uint32_t r;
    asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
    return r;
}

// All threads of the cluster: release this CTA's earlier writes (shared, distributed shared and
// global memory), wait for every CTA of the cluster, acquire theirs.
__device__ __forceinline__ void cluster_sync()
{
    asm volatile(
        "barrier.cluster.arrive.release.aligned;\n\t"
        "barrier.cluster.wait.acquire.aligned;" ::: "memory");
}

// The round barrier: the cluster barrier, or the CTA barrier when the cluster is one CTA (its
// partials then stay in its own shared memory, which the CTA barrier orders).
__device__ __forceinline__ void round_sync(int cs)
{
    if (cs == 1)
        __syncthreads();
    else
        cluster_sync();
}

// Shared-memory address of the same location in CTA `rank` of the cluster.
__device__ __forceinline__ uint32_t map_rank(uint32_t addr, uint32_t rank)
{
    uint32_t r;
    asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(addr), "r"(rank));
    return r;
}

__device__ __forceinline__ void st_cluster_u64(uint32_t addr, unsigned long long v)
{
    asm volatile("st.shared::cluster.u64 [%0], %1;" ::"r"(addr), "l"(v) : "memory");
}

// A stored unit word: SMALL tables hold the exact fp32 value of the unit (every unit is below 2^23),
// others the int32 unit. Bit 31 of column 0 marks a load-time duplicate and is cleared by the caller.
template <bool SMALL>
__device__ __forceinline__ float unit_f32(uint32_t w)
{
    return SMALL ? __uint_as_float(w) : __int2float_rn((int32_t)w);
}

template <bool SMALL>
__device__ __forceinline__ double unit_f64(uint32_t w)
{
    return SMALL ? (double)__uint_as_float(w) : __int2double_rn((int32_t)w);
}

template <bool SMALL>
__device__ __forceinline__ long long unit_i64(uint32_t w)
{
    return SMALL ? (long long)__float2int_rz(__uint_as_float(w)) : (long long)(int32_t)w;
}

template <bool SMALL>
__device__ __forceinline__ uint32_t stored_unit(int32_t u)
{
    if (!SMALL)
        return (uint32_t)u;
    const uint32_t sign = (uint32_t)u & 0x80000000u;
    return __float_as_uint((float)(u & 0x7fffffff)) | sign;
}

// This CTA's view of its slice and of the current prices.
template <int RT, bool UNI>
struct ResSlice {
    const uint32_t *U;      // unit words
    const double *V;        // values
    const int32_t *loff;    // CSR layout: slice-local option offset of each slice job (m + 1)
    int m;                  // jobs of the slice
    int stride;             // distance between the columns of one option (m_pad, or 1)
    int K;                  // uniform layout: options per job
    int jloc0;              // scenario-local index of the slice's first job
    int64_t gj0;            // global index of the slice's first job
    int R;
    float pf[ResCols<RT>::N];   // fp32 prices of the round
    const double *p64;          // fp64 prices of the round (shared memory)
    float e2;                   // 2E, +inf in exact mode
    bool exact;

    __device__ __forceinline__ int ucol0(int jj, int ob, int k) const
    {
        return UNI ? k * R * stride + jj : (ob + k) * R;
    }
    __device__ __forceinline__ int vslot(int jj, int ob, int k) const { return UNI ? k * stride + jj : ob + k; }
};

template <int RT, bool UNI, bool SMALL>
__device__ __forceinline__ float res_screen(const ResSlice<RT, UNI> &sl, int bu, double v, bool &dup)
{
    const uint32_t w0 = sl.U[bu];
    dup = (w0 >> 31) != 0;
    float q = -screen_value(v);
    q = __fmaf_rn(sl.pf[0], unit_f32<SMALL>(w0 & 0x7fffffffu), q);
#pragma unroll
    for (int r = 1; r < ResCols<RT>::N; ++r) {
        if (RT == 0 && r >= sl.R)
            break;
        q = __fmaf_rn(sl.pf[r], unit_f32<SMALL>(sl.U[bu + r * sl.stride]), q);
    }
    return q;
}

template <int RT, bool UNI, bool SMALL>
__device__ __forceinline__ double res_exact(const ResSlice<RT, UNI> &sl, int bu, double v)
{
    double s = -v;
#pragma unroll
    for (int r = 0; r < ResCols<RT>::N; ++r) {
        if (RT == 0 && r >= sl.R)
            break;
        uint32_t w = sl.U[bu + r * sl.stride];
        if (r == 0)
            w &= 0x7fffffffu;
        s = __fma_rn(sl.p64[r], unit_f64<SMALL>(w), s);
    }
    return s;
}

// Per-lane accumulators of one evaluation.
template <int RT>
struct ResAcc {
    long long dem[ResCols<RT>::N];
    unsigned long long hash;
    double dual;          // sum of -s_min over the lane's jobs
    unsigned int resolved;
};

// Exact resolution of one job: the lexicographic minimum of (s, k) over its survivors (options
// with q <= thr that are not load-time duplicates; every non-duplicate option in exact mode).
// Lane-serial form: the calling lane scans the job's options in order.
template <int RT, bool UNI, bool SMALL>
__device__ __forceinline__ int res_resolve_lane(const ResSlice<RT, UNI> &sl, int jj, int ob, int K, float thr,
                                                double &s_out)
{
    long long best = 0x7fffffffffffffffLL;
    int bi = kIdxNone;
    double bs = 0.0;
    for (int k = 0; k < K; ++k) {
        const int bu = sl.ucol0(jj, ob, k);
        const double v = sl.V[sl.vslot(jj, ob, k)];
        bool dup;
        const float q = res_screen<RT, UNI, SMALL>(sl, bu, v, dup);
        if (dup || (!sl.exact && q > thr))
            continue;
        const double sc = res_exact<RT, UNI, SMALL>(sl, bu, v);
        const long long key = order_key(sc);
        if (key < best) {
            best = key;
            bi = k;
            bs = sc;
        }
    }
    s_out = bs;
    return bi;
}

// The same minimum computed by the whole warp: lanes take options k = lane, lane + 32, ... and a
// butterfly keeps the smallest (key, k). Every lane returns the answer.
template <int RT, bool UNI, bool SMALL>
__device__ __forceinline__ int res_resolve_warp(const ResSlice<RT, UNI> &sl, int jj, int ob, int K, float thr,
                                                double &s_out, int lane)
{
    long long best = 0x7fffffffffffffffLL;
    int bi = kIdxNone;
    double bs = 0.0;
    for (int k = lane; k < K; k += 32) {
        const int bu = sl.ucol0(jj, ob, k);
        const double v = sl.V[sl.vslot(jj, ob, k)];
        bool dup;
        const float q = res_screen<RT, UNI, SMALL>(sl, bu, v, dup);
        if (dup || (!sl.exact && q > thr))
            continue;
        const double sc = res_exact<RT, UNI, SMALL>(sl, bu, v);
        const long long key = order_key(sc);
        if (key < best) {
            best = key;
            bi = k;
            bs = sc;
        }
    }
#pragma unroll
    for (int d = 16; d >= 1; d >>= 1) {
        const long long ok = __shfl_xor_sync(FULL, best, d);
        const int oi = __shfl_xor_sync(FULL, bi, d);
        const double os = __shfl_xor_sync(FULL, bs, d);
        if (ok < best || (ok == best && oi < bi)) {
            best = ok;
            bi = oi;
            bs = os;
        }
    }
    s_out = bs;
    return bi;
}

// Best responses of the slice's jobs: lane = job. FINAL writes the selection outputs; otherwise the
// demand (and, when asked, fingerprint and dual sum) of the winners accumulate in acc. Ambiguous
// jobs are resolved by the whole warp one after the other when they are few, else each by its lane.
template <int RT, bool UNI, bool SMALL, bool FINAL>
__device__ void res_evaluate(const DevState &st, const ResSlice<RT, UNI> &sl, bool want_hash, bool want_min,
                             ResAcc<RT> &acc, int warp, int lane)
{
    const int R = RT ? RT : sl.R;
    for (int jb = warp * 32; jb < sl.m; jb += kResWarps * 32) {
        const int jj = jb + lane;
        const bool act = jj < sl.m;
        int ob = 0, K = act ? sl.K : 0;
        if (!UNI && act) {
            ob = sl.loff[jj];
            K = sl.loff[jj + 1] - ob;
        }
        float m1 = INFINITY, m2 = INFINITY;
        int i1 = 0;
#pragma unroll 4
        for (int k = 0; k < K; ++k) {
            bool dup;
            float q = res_screen<RT, UNI, SMALL>(sl, sl.ucol0(jj, ob, k), sl.V[sl.vslot(jj, ob, k)], dup);
            q = dup ? INFINITY : q;
            const bool better = q < m1;
            m2 = better ? m1 : fminf(m2, q);
            i1 = better ? k : i1;
            m1 = fminf(m1, q);
        }
        const float thr = __fadd_ru(m1, sl.e2);
        const bool amb = act && (sl.exact || !(m2 > thr));
        int w = i1;
        double s_w = 0.0;
        bool have_s = false;
        uint32_t amask = __ballot_sync(FULL, amb);
        if (__popc(amask) > 4) {
            if (amb) {
                const int bi = res_resolve_lane<RT, UNI, SMALL>(sl, jj, ob, K, thr, s_w);
                w = (bi == kIdxNone) ? i1 : bi;    // the option of m1 always survives; defensive only
                have_s = true;
                ++acc.resolved;
            }
        } else {
            while (amask) {
                const int cl = __ffs(amask) - 1;
                amask &= amask - 1;
                const int cob = __shfl_sync(FULL, ob, cl);
                const int cK = __shfl_sync(FULL, K, cl);
                const float cthr = __shfl_sync(FULL, thr, cl);
                double cs_w;
                const int bi = res_resolve_warp<RT, UNI, SMALL>(sl, jb + cl, cob, cK, cthr, cs_w, lane);
                if (lane == cl) {
                    w = (bi == kIdxNone) ? i1 : bi;
                    s_w = cs_w;
                    have_s = true;
                    ++acc.resolved;
                }
            }
        }
        if (!act)
            continue;
        const int bw = sl.ucol0(jj, ob, w);
#pragma unroll
        for (int r = 0; r < ResCols<RT>::N; ++r) {
            if (RT == 0 && r >= R)
                break;
            uint32_t u = sl.U[bw + r * sl.stride];
            if (r == 0)
                u &= 0x7fffffffu;
            acc.dem[r] += unit_i64<SMALL>(u);
        }
        if (want_hash)
            acc.hash += splitmix64_mix(((uint64_t)(uint32_t)(sl.jloc0 + jj) << 32) | (uint32_t)w);
        if (FINAL || want_min) {
            const double vw = sl.V[sl.vslot(jj, ob, w)];
            if (!have_s)
                s_w = res_exact<RT, UNI, SMALL>(sl, bw, vw);
            if (FINAL) {
                const int64_t gj = sl.gj0 + jj;
                st.sel[gj] = w;
                st.job_val[gj] = vw;
                st.job_min[gj] = s_w;
            } else {
                acc.dual += -s_w;
            }
        }
    }
}

// Wrapping sum over the warp of 64-bit words by three 32-bit hardware reductions of 22-bit chunks
// (a chunk sum over 32 lanes stays below 2^27); exact for the int64 demand, whose totals are below
// 2^63, and for the fingerprint, which wraps by definition.
__device__ __forceinline__ unsigned long long warp_sum_u64(unsigned long long v)
{
    const unsigned long long c0 = __reduce_add_sync(FULL, (unsigned)(v & 0x3fffffu));
    const unsigned long long c1 = __reduce_add_sync(FULL, (unsigned)((v >> 22) & 0x3fffffu));
    const unsigned long long c2 = __reduce_add_sync(FULL, (unsigned)(v >> 44));
    return c0 + (c1 << 22) + (c2 << 44);
}

// Prices of lambda (lanes c < R of warp 0 hold lambda_c, R <= 16): the fp64 and fp32 per-unit prices
// (the same values as the streaming path's) and the screen bound 2E, written to shared memory. E
// only has to bound the screen error from above, so it is computed in fp32 with every operation
// rounded up: p <= p32 (1 + 2^-23) + 2^-149, M = max|v| + sum_r p_r max u_r and
// E = (4R + 16) 2^-24 M + 2^-99, each replaced by an upper bound; no fp64 operation beyond the
// prices themselves. A price bound above 2^100, or M above 2^100, selects exact mode.
__device__ __forceinline__ void res_set_prices(double lam, double capd, float umax_up, float vmax_up, int R,
                                               int mode, bool exact_only, double *p64s, float *p32s, float *e2s,
                                               int lane)
{
    const bool mine = lane < R;
    const double p = mine ? effective_price(lam, capd, mode) : 0.0;
    const float p32 = __double2float_rn(p);
    const float p_up = __fadd_ru(__fmul_ru(p32, 1.0f + 0x1p-23f), 0x1p-149f);
    float term = mine ? __fmul_ru(p_up, umax_up) : 0.0f;
#pragma unroll
    for (int d = 8; d >= 1; d >>= 1)    // lanes 0 .. 15 hold the terms
        term = __fadd_ru(term, __shfl_xor_sync(FULL, term, d));
    const bool huge = __any_sync(FULL, mine && !(p_up <= 0x1p100f));
    if (mine) {
        p64s[lane] = p;
        p32s[lane] = p32;
    }
    if (lane == 0) {
        const float M = __fadd_ru(vmax_up, term);
        float e2 = INFINITY;
        if (!exact_only && !huge && M <= 0x1p100f)
            e2 = 2.0f * __fadd_ru(__fmul_ru(M, (4.0f * R + 16.0f) * 0x1p-24f), 0x1p-99f);
        *e2s = e2;
    }
}

template <int RT, bool UNI, bool SMALL>
__global__ void __launch_bounds__(kResThreads, ESP_RES_MIN_CTAS) k_resident(DevTable t, DevState st, ResPlan rp, SolveArgs a)
{
    extern __shared__ __align__(16) unsigned char smem[];
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int cs = rp.cs;
    const uint32_t rank = cluster_rank();
    const int s = blockIdx.x / cs;
    const int R = t.R, P = t.P, J = t.J, T = a.T;

    const ResLayout L = res_layout(R, rp.k, rp.m_pad, rp.n_cap, cs);
    double *Vs = reinterpret_cast<double *>(smem + L.vals);
    uint32_t *Us = reinterpret_cast<uint32_t *>(smem + L.units);
    int32_t *loff = reinterpret_cast<int32_t *>(smem + L.loff);
    unsigned long long *wpart = reinterpret_cast<unsigned long long *>(smem + L.wpart);
    unsigned long long *cpart = reinterpret_cast<unsigned long long *>(smem + L.cpart);
    double *p64s = reinterpret_cast<double *>(smem + L.prices);
    float *p32s = reinterpret_cast<float *>(smem + L.prices + kMaxR * 8);
    float *e2s = p32s + kMaxR;
    int *stops = reinterpret_cast<int *>(e2s + 1);

    // ---- this CTA's slice of scenario s into shared memory (once)
    const int32_t *cut = rp.cuts + (size_t)s * (cs + 1);
    const int j0 = cut[rank], m = cut[rank + 1] - cut[rank];
    const int64_t gj0 = (int64_t)s * J + j0;
    const int64_t o0 = t.job_off[gj0];
    const int n = (int)(t.job_off[gj0 + m] - o0);
    {
        const int32_t *gu = t.units + o0 * R;
        for (int i = threadIdx.x; i < n * R; i += kResThreads) {
            const int o = i / R, r = i - o * R;
            const uint32_t w = stored_unit<SMALL>(__ldg(gu + i));
            if (UNI)
                Us[((o % rp.k) * R + r) * rp.m_pad + o / rp.k] = w;
            else
                Us[i] = w;
        }
        for (int o = threadIdx.x; o < n; o += kResThreads) {
            const double v = __ldg(t.values + o0 + o);
            if (UNI)
                Vs[(o % rp.k) * rp.m_pad + o / rp.k] = v;
            else
                Vs[o] = v;
        }
        if (!UNI)
            for (int jj = threadIdx.x; jj <= m; jj += kResThreads)
                loff[jj] = (int32_t)(t.job_off[gj0 + jj] - o0);
    }

    // ---- price state: warp 0 of every CTA holds lambda_c, C_c and max u_c in lane c
    const size_t sp = (size_t)s * P;
    double lam = 0.0, capd = 1.0;
    long long cap = 1;
    float umax_up = 0.0f;
    const float vmax_up = __double2float_ru(st.vmax[s]);
    if (warp == 0) {
        if (lane < R) {
            lam = st.lam[sp + lane];
            cap = t.cap[sp + lane];
            capd = (double)cap;
            umax_up = __int2float_ru(st.umax[(size_t)s * R + lane]);
        }
        res_set_prices(lam, capd, umax_up, vmax_up, R, a.mode, a.exact_only != 0, p64s, p32s, e2s, lane);
        if (lane == 0)
            *stops = 0;
    }
    // every CTA of the cluster is running (its shared memory may be written by peers from here on)
    // and this CTA's slice and prices are in place
    cluster_sync();

    ResSlice<RT, UNI> sl;
    sl.U = Us;
    sl.V = Vs;
    sl.loff = loff;
    sl.m = m;
    sl.stride = UNI ? rp.m_pad : 1;
    sl.K = rp.k;
    sl.jloc0 = j0;
    sl.gj0 = gj0;
    sl.R = R;
    sl.p64 = p64s;

    const bool want_hash = st.hash_trace != nullptr;
    const bool want_min = st.dual_trace != nullptr;
    ResAcc<RT> acc;
    acc.resolved = 0;
    int rounds = 0, status = 0, converged = 0;
    double best_dual = INFINITY;

    // Every CTA meets the same 1 + T + 1 cluster barriers whatever the data: once the stopping rule
    // (or a non-finite price) ends the scenario, the remaining rounds skip their work but still
    // meet the barrier, so no data-dependent decision can leave a peer waiting.
    bool stopped = false;
    for (int round = 0; round < T; ++round) {
        const int par = round & 1;
        if (!stopped) {
            // 1. best responses at the round's prices
#pragma unroll
            for (int r = 0; r < ResCols<RT>::N; ++r) {
                sl.pf[r] = (r < R) ? p32s[r] : 0.0f;
                acc.dem[r] = 0;
            }
            sl.e2 = *e2s;
            sl.exact = !(sl.e2 < INFINITY);
            acc.hash = 0ull;
            acc.dual = 0.0;
            res_evaluate<RT, UNI, SMALL, false>(st, sl, want_hash, want_min, acc, warp, lane);

            // 2. warp sums, then (after the barrier) the CTA partial in warp order
#pragma unroll
            for (int r = 0; r < ResCols<RT>::N; ++r) {
                if (RT == 0 && r >= R)
                    break;
                const long long v = (long long)warp_sum_u64((unsigned long long)acc.dem[r]);
                if (lane == 0)
                    wpart[warp * kResCols + r] = (unsigned long long)v;
            }
            if (want_hash) {
                const long long h = (long long)warp_sum_u64(acc.hash);
                if (lane == 0)
                    wpart[warp * kResCols + kColHash] = (unsigned long long)h;
            }
            if (want_min) {
                const double d = warp_sum_fixed(acc.dual);
                if (lane == 0)
                    wpart[warp * kResCols + kColDual] = (unsigned long long)__double_as_longlong(d);
            }
        }
        __syncthreads();

        // 3. the CTA partial into buffer (round & 1) of every CTA of the cluster
        if (!stopped && warp == 0) {
            const int c = lane;
            const bool live = c < R || (c == kColHash && want_hash) || (c == kColDual && want_min);
            if (live) {
                unsigned long long tot = 0ull;
                if (c == kColDual) {
                    double d = 0.0;
                    for (int w = 0; w < kResWarps; ++w)
                        d += __longlong_as_double((long long)wpart[w * kResCols + c]);
                    tot = (unsigned long long)__double_as_longlong(d);
                } else {
#pragma unroll
                    for (int w = 0; w < kResWarps; ++w)
                        tot += wpart[w * kResCols + c];
                }
                const uint32_t slot = smem_u32(cpart + ((size_t)par * cs + rank) * kResCols + c);
                for (int rk = 0; rk < cs; ++rk)
                    st_cluster_u64(map_rank(slot, (uint32_t)rk), tot);
            }
        }
        round_sync(cs);

        // 4. every CTA: the scenario's totals in rank order, then Eq. price_update
        if (!stopped && warp == 0) {
            const int c = lane;
            const unsigned long long *cp = cpart + (size_t)par * cs * kResCols;
            long long Uc = 0;
            if (c < R) {
#pragma unroll
                for (int rk = 0; rk < kResMaxCluster; ++rk)   // independent loads, summed in rank order
                    if (rk < cs)
                        Uc += (long long)cp[rk * kResCols + c];
            }
            const bool lead = rank == 0;
            if (want_min) {
                double d = 0.0;
                if (c == 0)
                    for (int rk = 0; rk < cs; ++rk)
                        d += __longlong_as_double((long long)cp[rk * kResCols + kColDual]);
                const double lc = (c < R) ? ((a.mode == 1) ? lam : lam * capd) : 0.0;
                const double g = __shfl_sync(FULL, d, 0) + warp_sum_fixed(lc);
                if (g < best_dual)
                    best_dual = g;
                if (lead && lane == 0)
                    st.dual_trace[(size_t)s * (T + 1) + round] = g;
            }
            if (want_hash && lead && lane == 0) {
                unsigned long long h = 0ull;
                for (int rk = 0; rk < cs; ++rk)
                    h += cp[rk * kResCols + kColHash];
                st.hash_trace[(size_t)s * T + round] = h;
            }
            if (st.dem_trace && lead && c < R)
                st.dem_trace[((size_t)s * T + round) * P + c] = Uc;
            const double eta = step_size(a.eta0, a.step, round);
            const double nl = (c < R) ? price_step(lam, Uc, cap, capd, eta, a.mode) : 0.0;
            const bool bad = __any_sync(FULL, c < R && !isfinite(nl));
            bool stop;
            if (bad) {
                status = 2;    // the prices stay at the last finite lambda
                stop = true;
            } else {
                rounds = round + 1;
                if (st.time_trace && lead && lane == 0)
                    st.time_trace[(size_t)s * T + round] = global_ns();
                if (st.lam_trace && lead && c < R)
                    st.lam_trace[((size_t)s * (T + 1) + round + 1) * P + c] = nl;
                stop = false;
                if (a.tol > 0.0) {   // the stopping rule on the step just taken
                    const double dmax = warp_max((c < R) ? fabs(nl - lam) : 0.0);
                    const double amax = warp_max((c < R) ? fabs(lam) : 0.0);
                    stop = dmax <= a.tol * fmax(1.0, amax);
                }
                lam = nl;
                converged = stop ? 1 : 0;
                res_set_prices(lam, capd, umax_up, vmax_up, R, a.mode, a.exact_only != 0, p64s, p32s, e2s, lane);
            }
            if (lane == 0)
                *stops = stop ? 1 : 0;
        }
        __syncthreads();
        stopped = *stops != 0;
    }

    // ---- final evaluation at the last prices: selection, values, minimal reduced costs, demand
#pragma unroll
    for (int r = 0; r < ResCols<RT>::N; ++r) {
        sl.pf[r] = (r < R) ? p32s[r] : 0.0f;
        acc.dem[r] = 0;
    }
    sl.e2 = *e2s;
    sl.exact = !(sl.e2 < INFINITY);
    res_evaluate<RT, UNI, SMALL, true>(st, sl, false, true, acc, warp, lane);
#pragma unroll
    for (int r = 0; r < ResCols<RT>::N; ++r) {
        if (RT == 0 && r >= R)
            break;
        const long long v = (long long)warp_sum_u64((unsigned long long)acc.dem[r]);
        if (lane == 0 && v != 0)
            atomicAdd(st.U_final + sp + r, (unsigned long long)v);
    }
    const unsigned int nres = __reduce_add_sync(FULL, acc.resolved);
    if (lane == 0 && nres)
        atomicAdd(st.stats, (unsigned long long)nres);
    if (warp == 0 && rank == 0) {
        if (lane < R)
            st.lam[sp + lane] = lam;
        if (lane == 0) {
            st.rounds_run[s] = rounds;
            st.converged[s] = converged;
            st.status[s] = status;
            st.frozen[s] = (converged || status) ? 1 : 0;
            if (want_min)
                st.best_dual[s] = best_dual;
        }
    }
    // no CTA leaves while a peer may still write into its shared memory
    cluster_sync();
}

template <int RT, bool UNI, bool SMALL>
struct ResKernel {
    static void *fn() { return reinterpret_cast<void *>(&k_resident<RT, UNI, SMALL>); }
};

template <typename F>
auto res_dispatch(int R, bool uni, bool small, F &&f)
{
#define ESP_RES_CASE(RT)                                                                                  \
    if (uni && small) return f(ResKernel<RT, true, true>());                                              \
    if (uni) return f(ResKernel<RT, true, false>());                                                      \
    if (small) return f(ResKernel<RT, false, true>());                                                    \
    return f(ResKernel<RT, false, false>());
    switch (R) {
    case 4: { ESP_RES_CASE(4) }
    case 6: { ESP_RES_CASE(6) }
    case 8: { ESP_RES_CASE(8) }
    default: { ESP_RES_CASE(0) }
    }
#undef ESP_RES_CASE
}

cudaLaunchConfig_t res_config(const DevTable &t, const ResPlan &rp, int64_t smem, cudaStream_t stream,
                              cudaLaunchAttribute *attr)
{
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)t.S * (unsigned)rp.cs, 1, 1);
    cfg.blockDim = dim3(kResThreads, 1, 1);
    cfg.dynamicSmemBytes = (size_t)smem;
    cfg.stream = stream;
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = (unsigned)rp.cs;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cfg;
}

// Function attributes, set once per kernel at load time (never during a stream capture): the
// device's whole opt-in shared memory as the ceiling (each launch asks for its own amount) and
// clusters of up to 16 CTAs.
cudaError_t res_prepare(void *fn)
{
    int dev = 0, optin = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e == cudaSuccess)
        e = cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev);
    if (e == cudaSuccess)
        e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, optin);
    if (e == cudaSuccess)
        e = cudaFuncSetAttribute(fn, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
    return e;
}

}  // namespace

int64_t res_smem_bytes(int R, const ResPlan &rp)
{
    return res_layout(R, rp.k, rp.m_pad, rp.n_cap, rp.cs).bytes;
}

cudaError_t res_max_clusters(const DevTable &t, const ResPlan &rp, bool small, int *n)
{
    *n = 0;
    const int64_t smem = res_smem_bytes(t.R, rp);
    return res_dispatch(t.R, rp.k > 0, small, [&](auto k) -> cudaError_t {
        void *fn = decltype(k)::fn();
        cudaError_t e = res_prepare(fn);
        if (e != cudaSuccess)
            return e;
        cudaLaunchAttribute attr[1];
        cudaLaunchConfig_t cfg = res_config(t, rp, smem, nullptr, attr);
        return cudaOccupancyMaxActiveClusters(n, fn, &cfg);
    });
}

cudaError_t launch_resident(const DevTable &t, const DevState &st, const ResPlan &rp, const SolveArgs &a,
                            cudaStream_t stream)
{
    const int64_t smem = res_smem_bytes(t.R, rp);
    return res_dispatch(t.R, rp.k > 0, t.small_units != 0, [&](auto k) -> cudaError_t {
        void *fn = decltype(k)::fn();
        cudaLaunchAttribute attr[1];
        cudaLaunchConfig_t cfg = res_config(t, rp, smem, stream, attr);
        void *args[] = {(void *)&t, (void *)&st, (void *)&rp, (void *)&a};
        return cudaLaunchKernelExC(&cfg, fn, args);
    });
}

}  // namespace esp
