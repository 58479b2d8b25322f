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
#include "esp_pass.cuh"

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
        if (st.ver)
            st.ver[s] = 0u;
        if (st.work && s == 0)
            *st.work = 0u;
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
    int n = dispatch_shape(R, grouped, mode,
                           [&](auto k) -> int { return pass_kernels_ctas_per_sm<decltype(k)>(smem); });
    if (n > 0 && pass_f32_shape(R, grouped, mode)) {
        // the plan must also suit the instantiation that reads fp32 stage units
        const int m = pass_ctas_per_sm_f32(R, mode, smem);
        n = m < n ? m : n;
    }
    return n;
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
    if (t.il_f32)
        return launch_pass_f32(t, st, pl, a, round, kind, grid, smem, stream, pdl);
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
