// Kernel interfaces of the ESP solver library (internal; the public ABI is include/esp.h).
#pragma once

#include <cstdint>
#include <cuda_runtime.h>

#include "esp_common.h"

namespace esp {

struct DevTable {
    const int32_t *units;     // n_opt * R
    const double *values;     // n_opt
    const int64_t *job_off;   // S*J + 1
    const uint16_t *group;    // n_opt or nullptr
    const int64_t *cap;       // S * P
    int64_t n_opt;
    int32_t S, J, R, P, r_global, n_groups;
    int32_t small_units;      // 1 if every unit is below 2^23
    const int32_t *jmap;      // sorted layout: original global index of each job of this table; nullptr: identity
    // evaluation passes only: the table tile by tile, each tile's units then its values, the tile of
    // options [a, b) at byte a * (4R + 8) (one bulk copy per tile); nullptr: units and values apart
    const unsigned char *il;
    // 1: il holds each unit as the bit pattern of its fp32 value (exact: every unit is below 2^23),
    // the duplicate mark still the sign bit of column 0
    int32_t il_f32;
};

struct DevState {
    double *lam;              // S*P prices lambda
    double *p64;              // S*P per-unit prices (lambda, or lambda / C in NORMALIZED mode)
    float *p32;               // S*P the same rounded to fp32 (the screen's prices)
    float *ebound;            // S   screen error bound E of the current prices; +inf: exact evaluation
    unsigned long long *U;    // S*P demand of the round being evaluated (int64 two's complement)
    unsigned long long *U_final; // S*P demand of the final selection
    unsigned long long *hash; // S   selection fingerprint of the round being evaluated
    int32_t *sel;             // S*J final selection (local index)
    double *job_val;          // S*J value of the final choice
    double *job_min;          // S*J minimal reduced cost (final pass; every round when tracing the dual)
    int32_t *rounds_run;      // S
    int32_t *converged;       // S
    int32_t *status;          // S   0 or 2 (a price became non-finite)
    int32_t *frozen;          // S   1 once a scenario stopped (converged or non-finite)
    double *best_dual;        // S
    double *primal;           // S
    double *dual;             // S
    int32_t *feasible;        // S
    const double *vmax;       // S   max |v| of the scenario (load time)
    const int32_t *umax;      // S*R max unit of each stored column in the scenario (load time)
    unsigned int *err;        // device error word (DEV_ERR_*)
    unsigned long long *stats;  // [0] exact resolutions since the last reset, [1] duplicates marked at load
    unsigned int *arrive;     // S   warps of the current round pass that finished the scenario
    unsigned int *ver;        // S   persistent pass: price updates applied to the scenario (kVerStopped once stopped)
    unsigned int *work;       // 1   persistent pass: work items handed out
    double *lam_trace;        // S*(T+1)*P or nullptr
    long long *dem_trace;     // S*T*P or nullptr
    unsigned long long *hash_trace; // S*T or nullptr
    double *dual_trace;       // S*(T+1) or nullptr
    unsigned long long *time_trace; // S*T or nullptr: global timer when each round's update was applied
};

struct DevPlan {
    const TileDesc *tiles;
    const int32_t *warp_begin;  // n_warps + 1
    int32_t n_warps;
    int32_t tile_opt;
    int32_t uniform_k;          // > 0: every job has exactly this many options, a power of two <= 32
    int32_t runs_only;          // 1: every tile is a run of equal-size jobs or a chunk of a large job
    const int32_t *scen_warps;  // S warps owning tiles of each scenario; non-null: round passes update prices
    const int32_t *scen_tiles;  // S tiles of each scenario (the persistent pass counts arrivals in tiles)
    const int32_t *item_order;  // n_warps: the persistent pass's ranges in the order it hands them out
};

struct SolveArgs {
    double eta0;
    int32_t step, mode, T;
    double tol;
    uint32_t flags;
    int32_t exact_only;
    uint32_t wait_ms;         // limit of a bounded stage wait, ms of the global timer (kWaitLimitMs: 4 s)
    uint32_t hold_tx;         // test hook, 0 normally: extra bytes announced on the first stage of the first
                              // round pass (warp 0), so that stage's phase never completes and its waits time out
};

enum PassKind : int32_t { PASS_ROUND = 0, PASS_FINAL = 1 };

// A placement table in factored form (esp_load_placement): option (k, n) of job j, local index
// k * N + n, has the units of configuration k (columns r >= r_global priced per node n, as a group)
// and the value cfg_values[j*KC + k] - (double)(sens[j] *fp32 D[job_type[j]*NT + node_type[n]]).
// Warps own contiguous job ranges.
struct DevPlace {
    const int32_t *cfg_units;     // n_jobs * KC * R
    const double *cfg_values;     // n_jobs * KC
    const float *sens;            // n_jobs
    const int32_t *job_type;      // n_jobs
    const int32_t *node_type;     // N
    const float *D;               // NT * NT
    const uint32_t *cfg_dup;      // n_jobs: bit k = configuration k repeats an earlier one of its job
    const int32_t *warp_job;      // n_warps + 1: first job of each warp
    const int32_t *scen_warps;    // S warps owning jobs of each scenario; non-null: round passes update prices
    int32_t KC, N, NT, n_warps;
};

constexpr int kPlaceMaxKC = 32;
constexpr int kPlaceMaxN = 64;
constexpr int kPlaceMaxNT = 64;
constexpr int kPlaceWarps = 4;
constexpr int kPlaceResMaxPrices = 1024;   // S * P limit of the grid-resident placement solve
constexpr int kPlaceResWarps = 16;         // warps per CTA of the grid-resident placement solve
constexpr int kPlaceResJobs = 2;           // jobs per warp it holds in shared memory
constexpr int kPlaceResPricesPerThread = (kPlaceResMaxPrices + kPlaceResWarps * 32 - 1) / (kPlaceResWarps * 32);

// The grid-resident placement solve (k_place_res): one CTA of kPlaceResWarps warps per SM, each warp
// holding at most kPlaceResJobs jobs; warp w owns the jobs [warp_job[w], warp_job[w + 1]).
struct PlaceRes {
    unsigned long long *U3;     // 3 * S * P: the demand of round r in buffer r % 3
    unsigned int *bar;          // [0] barrier arrivals, [1] abort; zeroed before each launch
    const int32_t *warp_job;    // n_warps + 1
    int32_t n_warps, grid;
};

// Shared-memory layout of k_place_res (byte offsets): the CTA's demand, price state and per-scenario
// reductions, then per warp the gs scratch and its cached jobs.
struct PlaceResLayout {
    int u, lam, p64, capd, cap, p32, eb, flags, maxes, warps;
    int warp_bytes, job_bytes, job_units, job_ufs, job_vals, job_pens, cand;
    int total;
};

__host__ __device__ inline PlaceResLayout place_res_layout(int S, int P, int KC, int R)
{
    auto up16 = [](int x) { return (x + 15) & ~15; };
    PlaceResLayout L;
    const int SP = S * P;
    L.u = 0;
    L.lam = L.u + up16(SP * 8);
    L.p64 = L.lam + up16(SP * 8);
    L.capd = L.p64 + up16(SP * 8);
    L.cap = L.capd + up16(SP * 8);
    L.p32 = L.cap + up16(SP * 8);
    L.eb = L.p32 + up16(SP * 4);
    L.flags = L.eb + up16(S * 4);
    L.maxes = L.flags + up16(6 * S * 4);
    L.warps = L.maxes + up16(2 * S * 8);
    // per warp: gs (KC floats), 32 candidate slots, then per job: units, fp32 units, values and the
    // fp32 penalty of every node
    const int head = up16(KC * 4) + 32 * 4;
    L.cand = up16(KC * 4);
    L.job_units = head;
    L.job_ufs = head + up16(KC * R * 4);
    L.job_vals = head + 2 * up16(KC * R * 4);
    L.job_pens = head + 2 * up16(KC * R * 4) + up16(KC * 8);
    L.job_bytes = 2 * up16(KC * R * 4) + up16(KC * 8) + kPlaceMaxN * 4;
    L.warp_bytes = head + kPlaceResJobs * L.job_bytes;
    L.total = L.warps + kPlaceResWarps * L.warp_bytes;
    return L;
}

int place_res_smem_bytes(int S, int P, int KC, int R);
int place_res_ctas_per_sm(int S, int P, int KC, int R);   // 0 if it cannot run

// All rounds of a placement solve in one cooperative launch of pr.grid CTAs (at most one per SM).
// Zeroes pr.bar and pr.U3 first.
cudaError_t launch_place_res(const DevTable &t, const DevState &st, const DevPlace &pl, const SolveArgs &a,
                             const PlaceRes &pr, cudaStream_t stream);

// Dynamic shared memory and resident CTAs per SM of the placement kernel (0 if it cannot run).
int place_smem_bytes(int R, int P, int KC, int N, int NT);
int place_ctas_per_sm(int R, int P, int KC, int N, int NT);
cudaError_t launch_place(const DevTable &t, const DevState &st, const DevPlace &pl, const SolveArgs &a, int round,
                         PassKind kind, int grid, cudaStream_t stream);

// Plan of the cluster-resident kernel: one cluster of cs CTAs per scenario; CTA c of scenario s holds
// the scenario-local jobs [cuts[s*(cs+1) + c], cuts[s*(cs+1) + c + 1]) in shared memory.
struct ResPlan {
    const int32_t *cuts;
    int32_t cs;
    int32_t k;          // > 0: every job has k options (interleaved layout); 0: CSR layout
    int32_t m_pad;      // job slots of a slice, a multiple of 32
    int64_t n_cap;      // option slots of a slice (CSR layout)
};

// Instantiations of the per-warp evaluation kernel: general tables (the segmented scan over job
// offsets), uniform tables (every job the same power-of-two option count), and sorted layouts, whose
// tiles are all runs of equal-size jobs or chunks of large jobs (no job offsets, no segmented scan).
enum : int { kModeGeneral = 0, kModeUniform = 1, kModeRuns = 2 };

inline int pass_mode(const DevPlan &pl)
{
    return pl.uniform_k > 0 ? kModeUniform : pl.runs_only ? kModeRuns : kModeGeneral;
}

// Dynamic shared memory per CTA of the evaluation kernel.
int pass_smem_bytes(int R, bool grouped, int mode, int P, int tile_opt);

// Maximum resident CTAs per SM of the evaluation kernel for this table shape (0 if it cannot run).
int pass_ctas_per_sm(int R, bool grouped, int mode, int P, int tile_opt);

// Table shapes with an instantiation of the evaluation kernel that reads the units of its
// tile-interleaved stage as fp32 (DevTable::il_f32; esp_kernels_f32.cu).
inline bool pass_f32_shape(int R, bool grouped, int mode)
{
    return !grouped && (R == 4 || R == 6 || R == 8) && (mode == kModeUniform || mode == kModeRuns);
}
// Resident CTAs per SM of that instantiation (0: the shape has none, or it cannot run).
int pass_ctas_per_sm_f32(int R, int mode, int smem);
// The persistent pass (rounds 0 .. n_rounds - 1 in one cooperative launch, esp_pass.cuh) exists for
// the same shapes, reading fp32 stage units. Its dynamic shared memory per CTA, its resident CTAs per
// SM (0: no such kernel or it cannot run) and its launch (grid at most the co-resident CTAs; fused
// updates; n_rounds * pl.n_warps below 2^31; k_init resets its item counter and versions).
int pass_persist_smem_bytes(int R, int P, int tile_opt);
int pass_persist_ctas_per_sm(int R, int mode, int P, int tile_opt);
cudaError_t launch_pass_persist(const DevTable &t, const DevState &st, const DevPlan &pl, const SolveArgs &a,
                                int n_rounds, int grid, cudaStream_t stream);
// Launches it (pass_f32_shape must hold for the table and plan).
cudaError_t launch_pass_f32(const DevTable &t, const DevState &st, const DevPlan &pl, const SolveArgs &a, int round,
                            PassKind kind, int grid, int smem, cudaStream_t stream, bool pdl);

cudaError_t launch_validate(const DevTable &t, double *vmax, int32_t *umax, unsigned int *flags,
                            cudaStream_t stream);
// Marks every option that repeats an earlier option of its job (units, value and group equal) by
// setting the sign bit of its column-0 unit in `units` (the device copy of t.units).
// max_k: the table's largest option count (jobs above 1024 options stay unmarked).
cudaError_t launch_mark_duplicates(const DevTable &t, int32_t *units, unsigned long long *marked, cudaStream_t stream,
                                   int64_t max_k);

// Fills the sorted layout of a general table: job j of `sorted` (offsets sorted.job_off, original
// job sorted.jmap[j]) receives the options of that original job of `orig`, followed by padding
// options (units 0 with the duplicate mark, value 0) up to its padded size.
cudaError_t launch_gather_sorted(const DevTable &orig, const DevTable &sorted, int32_t *units, double *values,
                                 cudaStream_t stream);
// v' = values0 - Gamma (Eq. esp_score's Gamma term) for every option; flags VAL_PENALTY.
cudaError_t launch_apply_penalties(const DevTable &t, const double *values0, const int32_t *c_cur, const double *s_hat,
                                   const double *tau, double gamma0, double alpha, double *values, unsigned int *flags,
                                   cudaStream_t stream);
// Fills the tile-interleaved copy `il` of table t (t.il's layout) for the n_tiles tiles of a plan;
// f32: units as fp32 bit patterns (DevTable::il_f32).
cudaError_t launch_interleave(const DevTable &t, const TileDesc *tiles, int64_t n_tiles, unsigned char *il,
                              bool f32, cudaStream_t stream);
// Clears every duplicate mark of a units array.
cudaError_t launch_clear_marks(int32_t *units, int64_t n_opt, int R, cudaStream_t stream);
cudaError_t launch_init(const DevTable &t, const DevState &st, const SolveArgs &a, const double *lambda0,
                        cudaStream_t stream);
// pdl: launch as a programmatic dependent of the previous kernel on the stream (the pass stages its
// first tiles before waiting for that kernel); only when the previous operation is a kernel.
cudaError_t launch_pass(const DevTable &t, const DevState &st, const DevPlan &pl, const SolveArgs &a,
                        int round, PassKind kind, int grid, cudaStream_t stream, bool pdl = false);
cudaError_t launch_update(const DevTable &t, const DevState &st, const SolveArgs &a, int round,
                          cudaStream_t stream);
// Dynamic shared memory of one resident CTA, and the clusters of the resident kernel that can be
// resident at once (0: the shape cannot run; needs the device). res_max_clusters also sets the
// kernel's function attributes and must run (at load time) before its first launch.
int64_t res_smem_bytes(int R, const ResPlan &rp);
cudaError_t res_max_clusters(const DevTable &t, const ResPlan &rp, bool small_units, int *n);
// init must have run; writes everything the final pass and the price updates of the streaming path
// write (prices, selection, values, minimal reduced costs, final demand, counters, traces).
cudaError_t launch_resident(const DevTable &t, const DevState &st, const ResPlan &rp, const SolveArgs &a,
                            cudaStream_t stream);
cudaError_t launch_objectives(const DevTable &t, const DevState &st, const SolveArgs &a, cudaStream_t stream);

}  // namespace esp
