// Host tile planner of the ESP solver (internal).
#pragma once

#include <cstdint>
#include <vector>

#include "esp_common.h"

namespace esp {

struct Plan {
    std::vector<TileDesc> tiles;
    std::vector<int32_t> warp_begin;  // n_warps + 1
    int32_t n_warps = 0;
    int32_t tile_opt = 0;
};

// Splits the jobs of a CSR table (offsets job_off[0 .. S*J]) into at most max_warps contiguous
// warp ranges of about equal option counts (cut at job boundaries), and each range into tiles of
// whole jobs of one scenario with at most tile_opt options; a job with more than tile_opt options
// becomes consecutive chunks of one warp. Returns false on inconsistent offsets.
bool plan_tiles(const int64_t *job_off, int32_t S, int32_t J, int32_t tile_opt, int32_t max_warps, Plan &out);

// Checks a plan against the table: every job covered exactly once and in order, chunks complete,
// every tile inside the table. Returns false on the first violation.
bool check_plan(const int64_t *job_off, int32_t S, int32_t J, const Plan &p);

// Slices of the cluster-resident kernel: every scenario's jobs split into cs contiguous runs of about
// equal option counts, run c starting at the first job whose first option lies at least
// floor(c * N_s / cs) options into the scenario (N_s = options of scenario s).
struct ResShape {
    int32_t cs = 0;
    int32_t m_max = 0;                // most jobs in one slice
    int64_t n_max = 0;                // most options in one slice
    std::vector<int32_t> cuts;        // S * (cs + 1) scenario-local job indices
};

// Fills out for cs CTAs per scenario. Returns false on inconsistent offsets.
bool plan_resident(const int64_t *job_off, int32_t S, int32_t J, int32_t cs, ResShape &out);

}  // namespace esp
