// Host tile planner: static work split of one evaluation pass over tiles and warps.
#include "esp_plan.h"

#include <algorithm>

namespace esp {

// Estimated cost of evaluating a tile, in SM cycles of one warp, from clock64 probes of the pass on
// GB300. A tile costs a fixed part (stage wait, copy issue, bookkeeping) plus one warp-wide step per
// "row": 128 options four per lane for uniform runs and chunks of large jobs (a run of jobs with K =
// 4m options gives each job 2^ceil(log2 m) lanes, so 32 / that many jobs share a row), 32 options
// one per lane otherwise; closing a chunked job adds its cross-warp reduction and winner read.
static int64_t tile_rows(const TileDesc &d)
{
    if (d.flags & TILE_BIG)
        return (d.n_opt + 127) / 128;
    if ((d.flags & TILE_RUN) && tile_run_k(d.flags) >= 4) {
        const int m = tile_run_k(d.flags) / 4;
        int lanes = 1;
        while (lanes < m)
            lanes <<= 1;
        const int per_row = 32 / lanes;
        return (d.n_job + per_row - 1) / per_row;
    }
    return (d.n_opt + 31) / 32;
}

static int64_t tile_cost(const TileDesc &d)
{
    return 1050 + 1650 * tile_rows(d) + ((d.flags & TILE_BIG_LAST) ? 850 : 0);
}

bool plan_tiles(const int64_t *off, int32_t S, int32_t J, int32_t tile_opt, int32_t max_warps, Plan &out,
                const int32_t *scen, const int32_t *runk)
{
    out.tiles.clear();
    out.warp_begin.clear();
    out.tile_opt = tile_opt;
    const int64_t n_jobs = (int64_t)S * J;
    if (tile_opt < 32 || (tile_opt & 31) || max_warps < 1)
        return false;
    if (n_jobs == 0) {
        out.n_warps = 0;
        out.warp_begin.push_back(0);
        return true;
    }
    const int64_t total = off[n_jobs];
    if (off[0] != 0 || total < n_jobs)
        return false;
    for (int64_t j = 0; j < n_jobs; ++j)   // every job needs at least one option
        if (off[j + 1] <= off[j])
            return false;

    // 1. tiles in job order: whole jobs of one scenario (and one run) up to tile_opt options, or the
    //    chunks of a job larger than a tile. Without scen, job j belongs to scenario j / J, tracked
    //    incrementally (s_cur, s_end) instead of dividing per job.
    out.tiles.reserve((size_t)std::min<int64_t>(n_jobs, total / std::max(1, tile_opt / 4) + S + 1));
    int32_t s_cur = 0;
    int64_t s_end = J;
    int64_t j = 0;
    while (j < n_jobs) {
        while (!scen && j >= s_end) {
            ++s_cur;
            s_end += J;
        }
        const int32_t s = scen ? scen[j] : s_cur;
        const int64_t K = off[j + 1] - off[j];
        if (K > tile_opt || (runk && runk[j] > kPassRunMaxK)) {
            const int64_t nch = (K + tile_opt - 1) / tile_opt;
            for (int64_t c = 0; c < nch; ++c) {
                TileDesc d;
                d.opt_begin = off[j] + c * tile_opt;
                d.job_begin = j;
                d.n_opt = (int32_t)std::min<int64_t>(tile_opt, K - c * tile_opt);
                d.n_job = (c == 0) ? 1 : 0;
                d.scenario = s;
                d.flags = TILE_BIG | (c == 0 ? TILE_BIG_FIRST : 0u) | (c == nch - 1 ? TILE_BIG_LAST : 0u);
                out.tiles.push_back(d);
            }
            ++j;
            continue;
        }
        const int64_t opt0 = off[j];
        const int32_t rk = runk ? runk[j] : 0;
        int64_t jj = j;
        const int64_t jlim = scen ? n_jobs : std::min<int64_t>(n_jobs, s_end);
        while (jj < jlim && (!scen || scen[jj] == s) && (!runk || runk[jj] == rk) && off[jj + 1] - opt0 <= tile_opt)
            ++jj;
        TileDesc d;
        d.opt_begin = opt0;
        d.job_begin = j;
        d.n_opt = (int32_t)(off[jj] - opt0);
        d.n_job = (int32_t)(jj - j);
        d.scenario = s;
        d.flags = rk > 0 ? tile_run_flags(rk) : 0u;
        out.tiles.push_back(d);
        j = jj;
    }

    // 2. warps: contiguous tile ranges of about equal estimated cost, at least one full tile of work
    //    per warp; a range never starts inside the chunks of a large job (its state is per warp)
    const int64_t n_tiles = (int64_t)out.tiles.size();
    std::vector<int64_t> pre(n_tiles + 1, 0);
    for (int64_t k = 0; k < n_tiles; ++k)
        pre[k + 1] = pre[k] + tile_cost(out.tiles[k]);
    const int64_t full = 1050 + 1650;     // one row
    const int64_t want = (pre[n_tiles] + full - 1) / full;
    const int32_t W = (int32_t)std::min<int64_t>(std::min<int64_t>(max_warps, std::max<int64_t>(1, want)), n_tiles);
    out.warp_begin.assign(W + 1, 0);
    out.warp_begin[W] = (int32_t)n_tiles;
    for (int32_t w = 1; w < W; ++w) {
        const int64_t target = (int64_t)((__int128)pre[n_tiles] * w / W);
        int64_t k = std::lower_bound(pre.begin(), pre.end(), target) - pre.begin();
        if (k > 0 && target - pre[k - 1] < pre[k] - target)   // the nearer tile boundary
            --k;
        if (k < n_tiles && (out.tiles[k].flags & TILE_BIG) && !(out.tiles[k].flags & TILE_BIG_FIRST)) {
            int64_t a = k, b = k;                            // the chunked job's first tile, the next job's
            while (!(out.tiles[a].flags & TILE_BIG_FIRST))
                --a;
            while (b < n_tiles && (out.tiles[b].flags & TILE_BIG) && !(out.tiles[b].flags & TILE_BIG_FIRST))
                ++b;
            k = (target - pre[a] < pre[b] - target) ? a : b;
        }
        k = std::min<int64_t>(std::max<int64_t>(k, out.warp_begin[w - 1]), n_tiles);
        out.warp_begin[w] = (int32_t)k;
    }
    out.n_warps = W;
    return true;
}

bool check_plan(const int64_t *off, int32_t S, int32_t J, const Plan &p, const int32_t *scen,
                const int32_t *runk)
{
    auto scen_of = [&](int64_t j) -> int64_t { return scen ? scen[j] : j / J; };
    const int64_t n_jobs = (int64_t)S * J;
    if ((int32_t)p.warp_begin.size() != p.n_warps + 1)
        return false;
    if (p.warp_begin.front() != 0 || p.warp_begin.back() != (int32_t)p.tiles.size())
        return false;
    for (int32_t w = 0; w < p.n_warps; ++w)
        if (p.warp_begin[w] > p.warp_begin[w + 1])
            return false;
    int64_t next_job = 0;
    int64_t big_next_opt = -1;  // expected opt_begin of the next chunk of an open big job
    for (const TileDesc &d : p.tiles) {
        if (d.n_opt < 1 || d.n_opt > p.tile_opt)
            return false;
        if (d.scenario < 0 || d.scenario >= S)
            return false;
        if (d.flags & TILE_BIG) {
            const int64_t j = d.job_begin;
            if (d.flags & TILE_BIG_FIRST) {
                if (big_next_opt >= 0 || j != next_job || d.opt_begin != off[j] || d.n_job != 1)
                    return false;
            } else if (d.opt_begin != big_next_opt || d.n_job != 0 || j != next_job) {
                return false;
            }
            if (scen_of(j) != d.scenario || d.opt_begin + d.n_opt > off[j + 1])
                return false;
            if (d.flags & TILE_BIG_LAST) {
                if (d.opt_begin + d.n_opt != off[j + 1])
                    return false;
                big_next_opt = -1;
                next_job = j + 1;
            } else {
                if (d.n_opt != p.tile_opt)
                    return false;
                big_next_opt = d.opt_begin + d.n_opt;
            }
        } else {
            if (big_next_opt >= 0 || d.job_begin != next_job || d.n_job < 1)
                return false;
            const int64_t j1 = d.job_begin + d.n_job;
            if (j1 > n_jobs || d.opt_begin != off[d.job_begin] || d.opt_begin + d.n_opt != off[j1])
                return false;
            if (!scen) {   // a contiguous range lies in one scenario iff its ends do
                if (scen_of(d.job_begin) != d.scenario || scen_of(j1 - 1) != d.scenario)
                    return false;
            }
            if (scen || runk) {
                for (int64_t j = d.job_begin; j < j1; ++j) {
                    if (scen && scen[j] != d.scenario)
                        return false;
                    if (d.flags & TILE_RUN) {
                        const int k = tile_run_k(d.flags);
                        if (!runk || runk[j] != k || off[j + 1] - off[j] != k || k > kPassRunMaxK)
                            return false;
                    } else if (runk && runk[j] != 0) {
                        return false;
                    }
                }
            } else if (d.flags & TILE_RUN) {
                return false;
            }
            if ((d.flags & TILE_RUN) && (d.opt_begin & 3) != 0 && tile_run_k(d.flags) >= 4)
                return false;   // a run of 4m-option jobs starts on a 4-option boundary
            next_job = j1;
        }
    }
    return big_next_opt < 0 && next_job == n_jobs;
}

bool plan_resident(const int64_t *off, int32_t S, int32_t J, int32_t cs, ResShape &out)
{
    out.cs = cs;
    out.m_max = 0;
    out.n_max = 0;
    out.cuts.assign((size_t)S * (cs + 1), 0);
    if (cs < 1 || S < 1 || J < 1)
        return false;
    for (int32_t s = 0; s < S; ++s) {
        const int64_t *o = off + (int64_t)s * J;   // o[0 .. J]
        const int64_t N = o[J] - o[0];
        if (N < J)
            return false;
        int32_t *cut = out.cuts.data() + (size_t)s * (cs + 1);
        cut[0] = 0;
        cut[cs] = J;
        for (int32_t c = 1; c < cs; ++c) {
            const int64_t target = o[0] + (int64_t)((__int128)N * c / cs);
            int32_t j = (int32_t)(std::lower_bound(o, o + J, target) - o);
            cut[c] = std::max(j, cut[c - 1]);
        }
        for (int32_t c = 0; c < cs; ++c) {
            out.m_max = std::max(out.m_max, cut[c + 1] - cut[c]);
            out.n_max = std::max<int64_t>(out.n_max, o[cut[c + 1]] - o[cut[c]]);
        }
    }
    return true;
}

bool sort_layout(const int64_t *off, int32_t S, int32_t J, SortedLayout &out, int32_t run_max_k)
{
    const int32_t kmax = run_max_k;
    if (kmax < 4 || (kmax & 3))
        return false;
    const int64_t n_jobs = (int64_t)S * J;
    out.off.assign(1, 0);
    out.jmap.clear();
    out.scen.clear();
    out.runk.clear();
    if (n_jobs < 1 || n_jobs >= INT32_MAX)
        return false;
    out.off.reserve(n_jobs + 1);
    out.jmap.reserve(n_jobs);
    out.scen.reserve(n_jobs);
    out.runk.reserve(n_jobs);
    auto push = [&](int64_t j, int32_t s, int64_t kp, int32_t rk) {
        out.off.push_back(out.off.back() + kp);
        out.jmap.push_back((int32_t)j);
        out.scen.push_back(s);
        out.runk.push_back(rk);
    };
    std::vector<std::vector<int32_t>> bucket(kmax / 4 + 1);
    for (int32_t s = 0; s < S; ++s) {       // jobs of 3 .. kmax options, padded to 4m
        for (auto &b : bucket)
            b.clear();
        for (int64_t j = (int64_t)s * J; j < (int64_t)(s + 1) * J; ++j) {
            const int64_t K = off[j + 1] - off[j];
            if (K < 1)
                return false;
            if (K >= 3 && K <= kmax)
                bucket[(K + 3) / 4].push_back((int32_t)j);
        }
        for (int b = 1; b <= kmax / 4; ++b)
            for (int32_t j : bucket[b])
                push(j, s, 4 * b, 4 * b);
    }
    for (int32_t s = 0; s < S; ++s)         // large jobs, unpadded
        for (int64_t j = (int64_t)s * J; j < (int64_t)(s + 1) * J; ++j)
            if (off[j + 1] - off[j] > kmax)
                push(j, s, off[j + 1] - off[j], 0);
    for (int32_t s = 0; s < S; ++s)         // runs of 2- and 1-option jobs
        for (int64_t k = 2; k >= 1; --k)
            for (int64_t j = (int64_t)s * J; j < (int64_t)(s + 1) * J; ++j)
                if (off[j + 1] - off[j] == k)
                    push(j, s, k, (int32_t)k);
    return (int64_t)out.jmap.size() == n_jobs;
}

}  // namespace esp
