// Instantiations of the evaluation-pass kernels (esp_pass.cuh: the round pass and the persistent
// pass) whose stage holds units as fp32 bit patterns: the tile-interleaved copy of a table without a group column whose units are all below
// 2^23 (DevTable::il_f32), for R = 4, 6, 8 on uniform tables and sorted layouts. The fp32 value of
// such a unit is exact, so the screen reads the same numbers as the integer kernels compute by one
// conversion per unit; selections, demands and prices are identical. Its own translation unit, so
// that it compiles in parallel with esp_kernels.cu.

#include "esp_pass.cuh"

namespace esp {

namespace {

template <typename Fn>
auto dispatch_f32(int R, int mode, Fn &&f)
{
    if (mode == kModeUniform) {
        switch (R) {
        case 4: return f(PassKernels<4, false, kModeUniform, true>());
        case 6: return f(PassKernels<6, false, kModeUniform, true>());
        default: return f(PassKernels<8, false, kModeUniform, true>());
        }
    }
    switch (R) {
    case 4: return f(PassKernels<4, false, kModeRuns, true>());
    case 6: return f(PassKernels<6, false, kModeRuns, true>());
    default: return f(PassKernels<8, false, kModeRuns, true>());
    }
}

template <typename Fn>
auto dispatch_persist(int R, int mode, Fn &&f)
{
    if (mode == kModeUniform) {
        switch (R) {
        case 4: return f(PersistKernel<4, kModeUniform, true>());
        case 6: return f(PersistKernel<6, kModeUniform, true>());
        default: return f(PersistKernel<8, kModeUniform, true>());
        }
    }
    switch (R) {
    case 4: return f(PersistKernel<4, kModeRuns, true>());
    case 6: return f(PersistKernel<6, kModeRuns, true>());
    default: return f(PersistKernel<8, kModeRuns, true>());
    }
}

}  // namespace

int pass_persist_smem_bytes(int R, int P, int tile_opt)
{
    return kWarpsPerCta * (warp_smem(tile_opt, R, false, P, false).bytes + kPersistQueueBytes);
}

int pass_persist_ctas_per_sm(int R, int mode, int P, int tile_opt)
{
    if (!pass_f32_shape(R, false, mode))
        return 0;
    const int smem = pass_persist_smem_bytes(R, P, tile_opt);
    return dispatch_persist(R, mode, [&](auto k) -> int {
        using K = decltype(k);
        if (cudaFuncSetAttribute(K::fn(), cudaFuncAttributeMaxDynamicSharedMemorySize, smem) != cudaSuccess)
            return 0;
        int n = 0;
        if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, K::fn(), kWarpsPerCta * 32, smem) != cudaSuccess)
            return 0;
        return n;
    });
}

cudaError_t launch_pass_persist(const DevTable &t, const DevState &st, const DevPlan &pl, const SolveArgs &a,
                                int n_rounds, int grid, cudaStream_t stream)
{
    const int mode = pass_mode(pl);
    if (!t.il_f32 || !pass_f32_shape(t.R, t.group != nullptr, mode) || pl.scen_warps == nullptr)
        return cudaErrorInvalidValue;
    const int smem = pass_persist_smem_bytes(t.R, t.P, pl.tile_opt);
    return dispatch_persist(t.R, mode, [&](auto k) -> cudaError_t {
        return decltype(k)::launch(grid, smem, stream, t, st, pl, a, n_rounds);
    });
}

int pass_ctas_per_sm_f32(int R, int mode, int smem)
{
    if (!pass_f32_shape(R, false, mode))
        return 0;
    return dispatch_f32(R, mode, [&](auto k) -> int { return pass_kernels_ctas_per_sm<decltype(k)>(smem); });
}

cudaError_t launch_pass_f32(const DevTable &t, const DevState &st, const DevPlan &pl, const SolveArgs &a, int round,
                            PassKind kind, int grid, int smem, cudaStream_t stream, bool pdl)
{
    const int mode = pass_mode(pl);
    if (t.group != nullptr || !pass_f32_shape(t.R, false, mode))
        return cudaErrorInvalidValue;
    const bool plain = kind == PASS_ROUND && st.hash_trace == nullptr && st.dual_trace == nullptr;
    dispatch_f32(t.R, mode, [&](auto k) -> int {
        decltype(k)::launch(plain, grid, smem, stream, t, st, pl, a, round, kind, pdl);
        return 0;
    });
    return cudaGetLastError();
}

}  // namespace esp
