// Shared host/device definitions of the ESP solver library (not part of the public ABI).
#pragma once

#include <cstdint>

#if defined(__CUDACC__)
#define ESP_HD __host__ __device__ __forceinline__
#else
#define ESP_HD inline
#endif

namespace esp {

// Tuning knobs (compile-time; the defaults are the measured best on GB300).
#ifndef ESP_STAGES
#define ESP_STAGES 2
#endif
#ifndef ESP_PREFETCH_TILES
#define ESP_PREFETCH_TILES 0
#endif
#ifndef ESP_UNIFORM4_TILE
#define ESP_UNIFORM4_TILE 128
#endif
#ifndef ESP_STAGE_DATA_BYTES
#define ESP_STAGE_DATA_BYTES 8192
#endif
#ifndef ESP_MIN_CTAS_UNIFORM
#define ESP_MIN_CTAS_UNIFORM 5
#endif
#ifndef ESP_MIN_CTAS_UNIFORM_NARROW
#define ESP_MIN_CTAS_UNIFORM_NARROW 6   // the same for R = 4 and R = 6 (80 registers, no spills)
#endif
#ifndef ESP_WARPS_PER_CTA
#define ESP_WARPS_PER_CTA 4
#endif
#ifndef ESP_GENERAL_TILE_MAX
#define ESP_GENERAL_TILE_MAX 128 // cap on the tile of general (CSR) tables (larger jobs become chunk tiles)
#endif
#ifndef ESP_MIN_CTAS_GENERAL
#define ESP_MIN_CTAS_GENERAL 4
#endif
#ifndef ESP_MIN_CTAS_RUNS
#define ESP_MIN_CTAS_RUNS 5       // register budget of the runs-only kernel (sorted layouts): 5 measured best
#endif
#ifndef ESP_V32_HW
#define ESP_V32_HW 0          // 1: fp64 -> fp32 of values by the conversion instruction (round to nearest)
#endif
#ifndef ESP_RES_WARPS
#define ESP_RES_WARPS 8       // warps per CTA of the cluster-resident kernel
#endif
#ifndef ESP_RES_MIN_CTAS
#define ESP_RES_MIN_CTAS 2    // register budget of the resident kernel: CTAs per SM it must allow
#endif
#ifndef ESP_BIGCHUNK4
#define ESP_BIGCHUNK4 1       // chunks of large jobs: four independent options per lane and step
#endif
#ifndef ESP_SORTED_LAYOUT
#define ESP_SORTED_LAYOUT 1   // general tables: evaluate a load-time layout sorted into runs of equal-size jobs
#endif
#ifndef ESP_I2F_COLS
#define ESP_I2F_COLS 16       // unit columns r < ESP_I2F_COLS use the int-to-float instruction
#endif

constexpr int kMaxR = 16;            // stored resource columns per option
constexpr int kWarpsPerCta = ESP_WARPS_PER_CTA;  // warps of a CTA; each warp owns its own stage ring
constexpr int kStages = ESP_STAGES;  // TMA stages per warp
constexpr int kPrefetchTiles = ESP_PREFETCH_TILES;  // L2 prefetch distance, in tiles of the warp
constexpr int kUniform4Tile = ESP_UNIFORM4_TILE;    // tile of the 4-options-per-lane path (0: largest)
constexpr int kMinCtasPerSm = ESP_MIN_CTAS_UNIFORM; // register budget of the uniform-K evaluation kernel
constexpr int kMinCtasPerSmNarrow = ESP_MIN_CTAS_UNIFORM_NARROW;  // ... for R = 4 and R = 6
constexpr int kMinCtasPerSmGeneral = ESP_MIN_CTAS_GENERAL;  // register budget of the general kernel
constexpr int kMinCtasPerSmRuns = ESP_MIN_CTAS_RUNS;        // ... of the runs-only kernel
constexpr int kStageDataBytes = ESP_STAGE_DATA_BYTES;  // option bytes (units + values [+ group]) of a full stage
// limit of a bounded stage wait of the evaluation passes, in milliseconds of the GPU's global timer
constexpr uint32_t kWaitLimitMs = 4000;

constexpr int kResWarps = ESP_RES_WARPS;
constexpr int kResMaxCluster = 16;   // CTAs per cluster of the resident kernel (16 is non-portable)
constexpr int kResCols = kMaxR + 2;  // words of a demand partial: R columns, fingerprint, dual sum

// Shared-memory layout of one CTA of the resident kernel: the CTA's slice of a scenario's table
// (uniform K: option k of slice job jj at slot k * m_pad + jj, so a warp reading one option of 32
// consecutive jobs touches 32 consecutive words; general: CSR order with local job offsets), the
// per-warp and per-cluster demand partials, and the prices of the current round.
struct ResLayout {
    int64_t vals, units, loff, wpart, cpart, prices, bytes;
};

ESP_HD ResLayout res_layout(int R, int K, int m_pad, long long n_cap, int cs)
{
    ResLayout L;
    const long long slots = K > 0 ? (long long)K * m_pad : n_cap;
    L.vals = 0;
    L.units = (slots * 8 + 15) & ~15LL;
    L.loff = L.units + ((slots * R * 4 + 15) & ~15LL);
    L.wpart = L.loff + (K > 0 ? 0 : (((long long)m_pad + 1) * 4 + 15) & ~15LL);
    L.cpart = L.wpart + (long long)kResWarps * kResCols * 8;
    L.prices = L.cpart + 2LL * cs * kResCols * 8;
    L.bytes = L.prices + kMaxR * 8 + kMaxR * 4 + 16;
    return L;
}

// Tile flags. A tile is a run of whole jobs of one scenario whose options are contiguous, or one
// chunk of a job with more options than a tile holds ("big" job).
enum : uint32_t {
    TILE_BIG = 1u,        // chunk of a big job
    TILE_BIG_FIRST = 2u,  // first chunk of its job
    TILE_BIG_LAST = 4u,   // last chunk of its job
    TILE_RUN = 8u,        // whole jobs that all have tile_run_k(flags) options (sorted layout)
};

ESP_HD int round16(int x) { return (x + 15) & ~15; }

// Options per job of a TILE_RUN tile (bits 8..19 of the flags).
ESP_HD int tile_run_k(uint32_t flags) { return (int)((flags >> 8) & 0xfffu); }
ESP_HD uint32_t tile_run_flags(int k) { return TILE_RUN | ((uint32_t)k << 8); }

// Largest padded job of the sorted layout (a multiple of 4): jobs of 3 .. kRunMaxK options are padded
// to a multiple of 4 and grouped into runs of equal size, which the per-warp pass evaluates as rows of
// whole jobs; larger jobs stay unpadded and are evaluated in chunks. (Measured on GB300 with the
// heavy-tailed table: padding the jobs of 129..256 options too, and reading their chunks four
// consecutive options per lane, was 2.5% and 7% slower than the unpadded, lane-strided chunks.)
#ifndef ESP_RUN_MAX_K
#define ESP_RUN_MAX_K 128
#endif
constexpr int kRunMaxK = ESP_RUN_MAX_K;
// Largest run tile of the per-warp pass (rows of whole jobs of up to 32 lanes x 4 options); a padded
// job above it is planned as chunks.
constexpr int kPassRunMaxK = 128;


struct TileDesc {
    int64_t opt_begin;    // first global option of the tile
    int64_t job_begin;    // global job index (s*J + j) of the first job starting in the tile, or of the big job
    int32_t n_opt;        // options in the tile (1 .. tile_opt)
    int32_t n_job;        // jobs starting in the tile (big chunks: 1 on the first chunk, else 0)
    int32_t scenario;
    uint32_t flags;
};
static_assert(sizeof(TileDesc) == 32, "TileDesc is 32 bytes");

// Options per tile for R stored columns: about kStageDataBytes of option data, a multiple of 32.
ESP_HD int tile_options(int R, bool grouped)
{
    int per = 4 * R + 8 + (grouped ? 2 : 0);
    int t = (kStageDataBytes / per) & ~31;
    return t < 32 ? 32 : t;
}

// Tile size for a table whose largest job has max_k options: large enough that every job of up to
// the maximum tile size stays whole (its exact resolution then reads the stage), at least 128
// options, and otherwise small so that more warps fit per SM.
ESP_HD int tile_options_for(int R, bool grouped, long long max_k, bool uniform4)
{
    const int cap = tile_options(R, grouped);
    if (uniform4)   // uniform jobs of 4..32 options: a fixed tile (the largest by default)
        return (kUniform4Tile > 0 && kUniform4Tile < cap) ? kUniform4Tile : cap;
    long long t = (max_k + 31) & ~31LL;
    if (t < 128)
        t = 128;
    if (ESP_GENERAL_TILE_MAX > 0 && t > ESP_GENERAL_TILE_MAX)
        t = ESP_GENERAL_TILE_MAX;
    return t > cap ? cap : (int)t;
}


// Byte layout of one stage. Every region starts 16-byte aligned and has room for the up-to-15
// bytes the bulk copy reads before and after its data to keep source and size 16-byte aligned.
struct StageLayout {
    int off, units, vals, grp, bytes;
};

ESP_HD StageLayout stage_layout(int tile_opt, int R, bool grouped, bool offsets)
{
    StageLayout L;
    L.off = 0;
    L.units = offsets ? round16((tile_opt + 1) * 8 + 32) : 0;   // uniform tables need no job offsets
    L.vals = L.units + round16(tile_opt * R * 4 + 32);
    L.grp = L.vals + round16(tile_opt * 8 + 32);
    L.bytes = L.grp + (grouped ? round16(tile_opt * 2 + 32) : 0);
    return L;
}

// Tile descriptors a warp keeps in shared memory: a ring refilled kDescBlock at a time, one block
// ahead of the block being issued.
constexpr int kDescRing = 16;
constexpr int kDescBlock = 8;
static_assert(kDescRing == 2 * kDescBlock, "two blocks in the descriptor ring");

// Per-warp shared memory: kStages stages, the tile-descriptor ring, the fp32 prices of the current
// scenario (grouped tables) and the stage barriers.
struct WarpSmem {
    int stage_bytes, descs, p32, bars, bytes;
};

ESP_HD WarpSmem warp_smem(int tile_opt, int R, bool grouped, int P, bool offsets)
{
    WarpSmem W;
    StageLayout L = stage_layout(tile_opt, R, grouped, offsets);
    W.stage_bytes = L.bytes;
    W.descs = kStages * L.bytes;          // the descriptor ring (32 bytes per tile)
    W.p32 = W.descs + 32 * kDescRing;
    W.bars = W.p32 + (grouped ? round16(P * 4) : 0);
    W.bytes = W.bars + 16 * kStages;
    return W;
}

// Persistent evaluation pass (every round in one cooperative launch): each warp keeps a queue of up to
// kPersistQueue taken work items (item, first tile, tiles, first virtual tile) in kPersistQueueBytes
// of shared memory after its WarpSmem.
constexpr int kPersistQueue = 8;
constexpr int kPersistMinTiles = 16;   // tiles per warp of the launch for the persistent pass by default
constexpr int kPersistQueueBytes = 4 * 4 * kPersistQueue;
// Price version of a scenario that stopped (converged or non-finite): every later round is released.
constexpr unsigned int kVerStopped = 0x7fffffffu;

// Device status words (bit flags in ctx error word).
enum : uint32_t {
    DEV_ERR_TIMEOUT = 1u,
    DEV_ERR_BAD_TABLE = 2u,
    DEV_ERR_PLAN = 4u,
};

// Load-time validation flags.
enum : uint32_t {
    VAL_UNITS_NEG = 1u,
    VAL_VALUE_NONFINITE = 2u,
    VAL_OFFSETS = 4u,
    VAL_GROUP_RANGE = 8u,
    VAL_CAPACITY = 16u,
    VAL_PENALTY = 32u,    // a current configuration outside its job, or a non-finite effective value
};

}  // namespace esp
