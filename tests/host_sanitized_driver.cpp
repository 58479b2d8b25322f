// Test driver for a build of the library's host code with AddressSanitizer and
// UndefinedBehaviorSanitizer (test infrastructure, compiled by tests/test_host_sanitized.py).
//
// Reads cases from a binary file of little-endian int64 words (doubles as their bit patterns):
//   n_cases, then per case: S, J, tile_opt, max_warps, cs, job offsets [S*J + 1]
//   then the host formulas: n, tau_base [n], beta, util, util_target, beta_max,
//                           R, capacity [R], Q, q_offsets [Q + 1], q_units [q_offsets[Q] * R], gamma
// and writes, as int64 words, per case:
//   the tile plan of the table:            ok, n_tiles, n_warps, 6 fields per tile, warp_begin [n_warps + 1]
//   the sorted layout:                     ok, then off [S*J + 1], jmap, scen, runk [S*J each]
//   the tile plan of the sorted layout:    ok, n_tiles, n_warps, tiles, warp_begin (only after a sorted layout)
//   the cluster-resident slices:           ok, m_max, n_max, n, cuts [n = S * (cs + 1)]
// then: status, tau_out [n] (bit patterns); status, c_eff [R].
// A plan that the planner accepts but its own check rejects exits with status 3.
#include <cstdint>
#include <cstdio>
#include <cstring>
#include <vector>

#include "esp.h"
#include "esp_plan.h"

namespace {

struct Reader {
    std::vector<int64_t> w;
    size_t at = 0;
    bool ok = true;
    int64_t next()
    {
        if (at >= w.size()) {
            ok = false;
            return 0;
        }
        return w[at++];
    }
    double next_f64()
    {
        const int64_t b = next();
        double d;
        std::memcpy(&d, &b, sizeof d);
        return d;
    }
};

struct Writer {
    std::vector<int64_t> w;
    void put(int64_t v) { w.push_back(v); }
    void put_f64(double d)
    {
        int64_t b;
        std::memcpy(&b, &d, sizeof b);
        w.push_back(b);
    }
};

void put_plan(Writer &out, bool ok, const esp::Plan &p)
{
    out.put(ok ? 1 : 0);
    if (!ok)
        return;
    out.put((int64_t)p.tiles.size());
    out.put(p.n_warps);
    for (const esp::TileDesc &d : p.tiles) {
        out.put(d.opt_begin);
        out.put(d.job_begin);
        out.put(d.n_opt);
        out.put(d.n_job);
        out.put(d.scenario);
        out.put((int64_t)d.flags);
    }
    for (int32_t v : p.warp_begin)
        out.put(v);
}

}  // namespace

int main(int argc, char **argv)
{
    if (argc != 3) {
        std::fprintf(stderr, "usage: %s cases.bin results.bin\n", argv[0]);
        return 2;
    }
    Reader in;
    {
        std::FILE *f = std::fopen(argv[1], "rb");
        if (!f)
            return 2;
        int64_t v;
        while (std::fread(&v, sizeof v, 1, f) == 1)
            in.w.push_back(v);
        std::fclose(f);
    }
    Writer out;
    const int64_t n_cases = in.next();
    for (int64_t c = 0; c < n_cases && in.ok; ++c) {
        const int32_t S = (int32_t)in.next(), J = (int32_t)in.next();
        const int32_t tile_opt = (int32_t)in.next(), max_warps = (int32_t)in.next(), cs = (int32_t)in.next();
        std::vector<int64_t> off((size_t)S * J + 1);
        for (int64_t &o : off)
            o = in.next();
        if (!in.ok)
            break;

        esp::Plan p;
        const bool planned = esp::plan_tiles(off.data(), S, J, tile_opt, max_warps, p);
        if (planned && !esp::check_plan(off.data(), S, J, p))
            return 3;
        put_plan(out, planned, p);

        esp::SortedLayout lay;
        const bool sorted = esp::sort_layout(off.data(), S, J, lay);
        out.put(sorted ? 1 : 0);
        if (sorted) {
            for (int64_t v : lay.off)
                out.put(v);
            for (int32_t v : lay.jmap)
                out.put(v);
            for (int32_t v : lay.scen)
                out.put(v);
            for (int32_t v : lay.runk)
                out.put(v);
            esp::Plan pr;
            const bool ok = esp::plan_tiles(lay.off.data(), S, J, tile_opt, max_warps, pr, lay.scen.data(),
                                            lay.runk.data());
            if (ok && !esp::check_plan(lay.off.data(), S, J, pr, lay.scen.data(), lay.runk.data()))
                return 3;
            put_plan(out, ok, pr);
        }

        esp::ResShape rs;
        const bool res = esp::plan_resident(off.data(), S, J, cs, rs);
        out.put(res ? 1 : 0);
        if (res) {
            out.put(rs.m_max);
            out.put(rs.n_max);
            out.put((int64_t)rs.cuts.size());
            for (int32_t v : rs.cuts)
                out.put(v);
        }
    }

    const int64_t n = in.next();
    std::vector<double> tau_base((size_t)(n > 0 ? n : 0)), tau((size_t)(n > 0 ? n : 0));
    for (double &t : tau_base)
        t = in.next_f64();
    const double beta = in.next_f64(), util = in.next_f64(), util_target = in.next_f64(), beta_max = in.next_f64();
    const int32_t R = (int32_t)in.next();
    std::vector<int64_t> cap((size_t)(R > 0 ? R : 0)), c_eff((size_t)(R > 0 ? R : 0));
    for (int64_t &v : cap)
        v = in.next();
    const int32_t Q = (int32_t)in.next();
    std::vector<int64_t> q_off((size_t)(Q >= 0 ? Q + 1 : 1));
    for (int64_t &v : q_off)
        v = in.next();
    std::vector<int32_t> q_units((size_t)(q_off.back() > 0 ? q_off.back() * R : 0));
    for (int32_t &v : q_units)
        v = (int32_t)in.next();
    const double gamma = in.next_f64();
    if (!in.ok)
        return 2;
    out.put(esp_adaptive_threshold(n, tau_base.data(), beta, util, util_target, beta_max, tau.data()));
    for (double t : tau)
        out.put_f64(t);
    out.put(esp_effective_capacity(R, cap.data(), Q, q_off.data(), q_units.empty() ? nullptr : q_units.data(),
                                   gamma, c_eff.data()));
    for (int64_t v : c_eff)
        out.put(v);

    std::FILE *f = std::fopen(argv[2], "wb");
    if (!f)
        return 2;
    const size_t wrote = std::fwrite(out.w.data(), sizeof(int64_t), out.w.size(), f);
    std::fclose(f);
    return wrote == out.w.size() ? 0 : 2;
}
