/*
 * esp_debug.h - helpers of the ESP solver library for tests: the host tile planner (no GPU code)
 * and counters of a context.
 */
#ifndef ESP_DEBUG_H
#define ESP_DEBUG_H

#include <stdint.h>

#include "esp.h"
#include "esp_iac.h"

#ifdef __cplusplus
extern "C" {
#endif

/* Counters of a loaded context: *resolutions = jobs whose fp32 screen was ambiguous and that were
 * resolved in fp64 since the last reset (all evaluation passes, including esp_evaluate), *marked =
 * options marked at load as exact duplicates of an earlier option of their job. Waits for the
 * context's stream; reset != 0 zeroes the resolution counter. */
esp_status esp_debug_stats(esp_ctx *ctx, int64_t *resolutions, int64_t *marked, int32_t reset);

/* Options per tile the evaluation pass uses for R stored columns (grouped != 0: a group column is
 * present). */
int32_t esp_debug_tile_options(int32_t R, int32_t grouped);

/* Runs the host tile planner on CSR offsets (host, S*J + 1 int64) for at most max_warps warps.
 * tiles: host buffer of tiles_cap * 8 int32 words receiving each tile as
 * {opt_begin lo, opt_begin hi, job_begin lo, job_begin hi, n_opt, n_job, scenario, flags};
 * warp_begin: host buffer of warps_cap + 1 int32. *n_tiles and *n_warps receive the counts.
 * Returns ESP_OK, ESP_ERR_INVALID_ARG for inconsistent offsets or a failed plan check, or
 * ESP_ERR_OOM when a buffer is too small (the counts are still written). */
esp_status esp_debug_plan(const int64_t *job_offsets, int32_t S, int32_t J, int32_t tile_opt, int32_t max_warps,
                          int32_t *tiles, int32_t tiles_cap, int32_t *warp_begin, int32_t warps_cap,
                          int32_t *n_tiles, int32_t *n_warps);

/* Sorted layout of a general table (jobs of varying size, no group column), as esp_load_options
 * builds it for the evaluation pass: per scenario the jobs of 3..256 options padded to a multiple
 * of 4 and ordered by padded size (this part first for every scenario), then per scenario the
 * larger jobs, then per scenario the 2-option and the 1-option jobs. Host buffers:
 *   off   S*J + 1 int64: padded option offsets in sorted order
 *   jmap  S*J int32: original global job index of each sorted job
 *   scen  S*J int32: scenario of each sorted job
 *   runk  S*J int32: options (padded) of the jobs of the sorted job's run, 0 for a large job
 * Returns ESP_ERR_INVALID_ARG for inconsistent offsets or more than 2^31 - 1 jobs. */
esp_status esp_debug_sort_layout(const int64_t *job_offsets, int32_t S, int32_t J, int64_t *off, int32_t *jmap,
                                 int32_t *scen, int32_t *runk);

/* esp_debug_plan for a sorted layout (the arrays esp_debug_sort_layout returns): tiles never mix
 * scenarios or runs, and a tile of a run has flag bit 3 set and its jobs' option count in bits 8..19
 * of its flags. Same buffers and errors as esp_debug_plan. */
esp_status esp_debug_plan_runs(const int64_t *off, const int32_t *scen, const int32_t *runk, int32_t S, int32_t J,
                               int32_t tile_opt, int32_t max_warps, int32_t *tiles, int32_t tiles_cap,
                               int32_t *warp_begin, int32_t warps_cap, int32_t *n_tiles, int32_t *n_warps);

/* enable = 0 makes later esp_load_options calls on this context evaluate general tables in their
 * original layout (the segmented path) instead of the sorted one; 1 restores the default. */
esp_status esp_debug_set_sorted_layout(esp_ctx *ctx, int32_t enable);

/* Programmatic dependent launch of the evaluation passes (each pass stages its first tiles while the
 * kernel before it finishes): mode -1 automatic (the library's choice per table), 0 off, 1 on. Takes
 * effect from the next solve; results are the same either way. */
esp_status esp_debug_set_pdl(esp_ctx *ctx, int32_t mode);

/* Warps of the evaluation pass planned by later loads, as a number of waves of resident CTAs
 * (1..8; 0 = the library's choice, two waves): more waves give smaller warp ranges that the hardware
 * schedules as CTAs finish. Results are the same for any setting. */
esp_status esp_debug_set_plan_waves(esp_ctx *ctx, int32_t waves);

/* Cluster size of the resident kernel (ESP_FLAG_RESIDENT) for the loaded table. force_cs: 0 keeps the
 * automatic choice; 1, 2, 4, 8 or 16 forces that many CTAs per scenario for later solves (the size must
 * fit the table). *cs receives the size solves use and *clusters how many such clusters the device
 * holds at once (either may be NULL). ESP_ERR_UNSUPPORTED: the table cannot run resident at all;
 * ESP_ERR_INVALID_ARG: force_cs is not a size that fits. */
esp_status esp_debug_resident(esp_ctx *ctx, int32_t force_cs, int32_t *cs, int32_t *clusters);

/* Failure-detection hook of the grid-resident placement solve (the bounded grid barrier): the next
 * esp_solve with ESP_FLAG_RESIDENT starts the barrier's arrival counter far short of its targets, so
 * no CTA passes the first barrier. Every CTA's wait gives up after its time limit (4 s of the GPU's
 * global timer) or when another CTA has given up; the solve returns ESP_ERR_TIMEOUT and the context
 * answers ESP_ERR_STATE from then on (destroy it; the device stays usable). One solve only.
 * ESP_ERR_UNSUPPORTED: no placement table is loaded, or it cannot run grid-resident. */
esp_status esp_debug_hold_barrier(esp_ctx *ctx);

/* Failure-detection hooks of the evaluation pass. esp_debug_set_wait_limit sets how long a bounded
 * wait of the pass's stage ring polls, in milliseconds of the GPU's global timer, before it gives up:
 * limit_ms = 0 restores the default (4000); a test sets a few to make a timeout short. esp_debug_hold_stage makes the next esp_solve's first round pass announce 16 more
 * bytes on the first stage of its first CTA (warp) than its copies bring, so that stage's barrier
 * phase never completes: no memory is accessed out of place, every wait on that phase runs out, and
 * the solve returns ESP_ERR_TIMEOUT; the context then answers ESP_ERR_STATE (destroy it; the device
 * stays usable). One solve only. */
esp_status esp_debug_set_wait_limit(esp_ctx *ctx, uint32_t limit_ms);
esp_status esp_debug_hold_stage(esp_ctx *ctx);

/* Allocation-failure injection (host side): the n-th next device allocation of this context (0: the
 * very next) reports ESP_ERR_OOM as a failed cudaMalloc would; n < 0 disarms it. */
esp_status esp_debug_fail_alloc(esp_ctx *ctx, int64_t n);

/* *kind receives how the loaded table is evaluated: 0 the per-warp pass with two bulk copies per tile
 * (units and values apart), 1 the per-warp pass with one bulk copy per tile (tile-interleaved table),
 * 2 the factored placement pass, 3 as 1 with the units of the interleaved table stored as fp32 (every
 * unit below 2^23, so each is exact; the screen then needs no conversion per unit). */
esp_status esp_debug_pass_kernel(esp_ctx *ctx, int32_t *kind);

/* Persistent pass: every round of a solve in one cooperative launch, each scenario's next round
 * released by its price update instead of a kernel boundary (tables whose interleaved tiles hold fp32
 * units; solves without per-pass events, fingerprint or dual trace). mode -1 (the default) uses it on
 * uniform tables with at least 16 tiles per warp of its launch, 0 never, 1 wherever the table can take
 * it; later solves of this context follow the mode. Results are identical either way.
 * esp_debug_persistent: *grid receives the CTAs of the persistent launch that a plain solve of the
 * loaded table uses under the current mode (0: one launch per round). */
esp_status esp_debug_set_persistent(esp_ctx *ctx, int32_t mode);
esp_status esp_debug_persistent(esp_ctx *ctx, int32_t *grid);
/* Waits of the persistent pass for a scenario's prices that had to poll since the last reset: *ns their
 * total duration in nanoseconds of the GPU's global timer (summed over warps), *waits their number.
 * Waits for the context's stream; reset != 0 zeroes both. */
esp_status esp_debug_persist_waits(esp_ctx *ctx, int64_t *ns, int64_t *waits, int32_t reset);

/* Profile of the last esp_load_options / esp_load_options_device of this context: ms[0..6] the host
 * milliseconds from its start until its uploads and validation were queued, until the sorted layout
 * was queued, until the occupancy of the pass kernels was known, until the pass was planned, until
 * the uploads, validation and duplicate marks were done, until the tiles, interleaved table and solve
 * state were queued, and until it returned; *mallocs and *frees the cudaMalloc and cudaFree calls it
 * made (a reload of a table of the same shape makes none). */
esp_status esp_debug_load_profile(esp_ctx *ctx, double *ms, int64_t *mallocs, int64_t *frees);

/* enable = 0 makes later loads keep integer units in the tile-interleaved table; 1 restores the
 * default (fp32 units where every unit is below 2^23 and the table has no group column, R = 4, 6 or 8,
 * uniform or sorted). Results are identical either way. */
esp_status esp_debug_set_stage_f32(esp_ctx *ctx, int32_t enable);

/* enable = 0 makes later loads keep the per-warp pass's table as separate unit and value arrays (two
 * bulk copies per tile); 1 restores the default, a tile-interleaved copy (each tile's units then its
 * values, one bulk copy per tile) wherever every tile allows it (esp_debug_pass_kernel then reports
 * 1). Results are identical either way. */
esp_status esp_debug_set_interleave(esp_ctx *ctx, int32_t enable);

/* Failure-detection hooks of the IAC predictor's tensor-core kernel (esp_iac.h). limit_ms bounds each
 * wait for an MMA group (in polls of at most 1 ms; 0 restores the default, about 4 s).
 * esp_iac_debug_hold_commit makes the next tensor-path launch leave its first MMA group in CTA 0's
 * first warpgroup uncommitted, so that warpgroup's wait runs out: no memory is accessed out of place,
 * the warpgroup then makes its barrier track every MMA still in flight, waits for them and leaves,
 * and esp_iac_synchronize answers ESP_ERR_TIMEOUT; the handle then answers ESP_ERR_STATE (destroy it;
 * the device stays usable). One launch only; ESP_ERR_UNSUPPORTED on the CUDA-core path. */
esp_status esp_iac_debug_set_wait_limit(esp_iac *m, uint32_t limit_ms);
esp_status esp_iac_debug_hold_commit(esp_iac *m);

#ifdef __cplusplus
}
#endif
#endif
