/*
 * esp_debug.h - host-only helpers of the ESP solver library for tests. They run no GPU code.
 */
#ifndef ESP_DEBUG_H
#define ESP_DEBUG_H

#include <stdint.h>

#include "esp.h"

#ifdef __cplusplus
extern "C" {
#endif

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

#ifdef __cplusplus
}
#endif
#endif
