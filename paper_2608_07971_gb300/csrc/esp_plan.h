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
// becomes consecutive chunks of one warp. scen (optional) gives each job's scenario (default j / J);
// runk (optional) gives each job the option count of its run in the sorted layout (0: not in a
// run): tiles never mix runs, and a tile of a run carries tile_run_flags(k). Returns false on
// inconsistent offsets.
bool plan_tiles(const int64_t *job_off, int32_t S, int32_t J, int32_t tile_opt, int32_t max_warps, Plan &out,
                const int32_t *scen = nullptr, const int32_t *runk = nullptr);

// Checks a plan against the table: every job covered exactly once and in order, chunks complete,
// every tile inside the table and inside one scenario (and one run). Returns false on the first
// violation.
bool check_plan(const int64_t *job_off, int32_t S, int32_t J, const Plan &p, const int32_t *scen = nullptr,
                const int32_t *runk = nullptr);

// Sorted layout of a general table (jobs of varying size, no group column), built at load time so
// that most jobs are evaluated as runs of equal size. Per scenario: the jobs of 3 .. kRunMaxK
// options, each padded with never-chosen options to a multiple of 4 and ordered by padded size
// (original order within a size); this part comes first for every scenario, so every run starts on
// a 4-option boundary. Then, per scenario, the jobs of more than kRunMaxK options, then the runs
// of 2-option and of 1-option jobs.
struct SortedLayout {
    std::vector<int64_t> off;    // S*J + 1 padded option offsets in sorted order
    std::vector<int32_t> jmap;   // sorted job -> original global job index
    std::vector<int32_t> scen;   // scenario of each sorted job
    std::vector<int32_t> runk;   // options (padded) of every job of the sorted job's run, 0 for a large job
};

// Returns false when the table is not eligible (more than 2^31 - 1 jobs, or inconsistent offsets).
// run_max_k: the largest padded job of the runs (a multiple of 4; the library uses kRunMaxK).
bool sort_layout(const int64_t *job_off, int32_t S, int32_t J, SortedLayout &out, int32_t run_max_k = kRunMaxK);



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
