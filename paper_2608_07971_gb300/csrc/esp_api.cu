// C ABI of the ESP solver (include/esp.h): context, table upload and validation, solve driver.
#include <cmath>
#include <cstdint>
#include <algorithm>
#include <chrono>
#include <cstring>
#include <new>
#include <vector>

#include <cuda_runtime.h>

#include "esp.h"
#include "esp_debug.h"
#include "esp_kernels.h"
#include "esp_place.h"
#include "esp_plan.h"

using namespace esp;

namespace {

struct GraphKey {
    double eta0 = 0, tol = 0;
    int32_t step = -1, mode = -1, T = -1;
    uint32_t flags = 0;
    const void *lt = nullptr, *dt = nullptr, *ht = nullptr, *gt = nullptr, *tt = nullptr;
    bool has_l0 = false;
    int res = -1;   // resident option in use, -1: streaming
    bool hold = false;
    bool persist = false;   // rounds in one persistent launch
    uint32_t hold_tx = 0, wait_ms = 0;
    uint64_t args = 0;      // hash of every kernel argument and launch shape of the solve
    bool operator==(const GraphKey &o) const
    {
        return eta0 == o.eta0 && tol == o.tol && step == o.step && mode == o.mode && T == o.T && flags == o.flags &&
               persist == o.persist && args == o.args &&
               lt == o.lt && dt == o.dt && ht == o.ht && gt == o.gt && tt == o.tt && has_l0 == o.has_l0 &&
               res == o.res &&
               hold == o.hold && hold_tx == o.hold_tx && wait_ms == o.wait_ms;
    }
};

template <typename T>
struct DevArr {
    T *p = nullptr;
    size_t n = 0;
};

}  // namespace

// The host plan of a load (option counts, sorted layout, tiles and warp ranges), kept for the next
// load of a table with the same shape and offsets.
struct PlanCache {
    bool valid = false;
    int32_t S = 0, J = 0, R = 0, P = 0, max_warps = 0, tile_opt = 0;
    bool grouped = false, sorted_enabled = false;
    std::vector<int64_t> off;
    int64_t min_k = 0, max_k = 0;
    bool sorted = false;
    esp::SortedLayout lay;
    esp::Plan plan;
};

struct esp_ctx {
    int device = 0;
    cudaStream_t stream = nullptr;
    int sm_count = 0;
    bool poisoned = false;
    bool loaded = false;
    bool solved = false;

    int32_t S = 0, J = 0, R = 0, P = 0, rg = 0, n_groups = 0;
    int64_t max_k = 0;   // largest option count of the loaded table
    int64_t n_opt = 0;
    int32_t small_units = 0;
    PlanCache pc;
    // device buffers of the loaded table and solve state (pointer, bytes); a reload hands them to
    // `pool`, from which the new table's allocations are served when the sizes fit
    std::vector<std::pair<void *, size_t>> table_bufs;
    std::vector<std::pair<void *, size_t>> pool;
    int32_t *units = nullptr;
    double *values = nullptr;
    int64_t *off = nullptr;
    // sorted layout of a general table (the evaluation pass reads it; outputs use jmap)
    bool sorted_enabled = ESP_SORTED_LAYOUT != 0;   // later loads build it (esp_debug_set_sorted_layout)
    int pdl_mode = -1;   // programmatic dependent launch of the passes: -1 automatic, 0 off, 1 on
    bool res_planned = false;   // resident options planned for the loaded table
    int plan_waves = 0;         // warps of the evaluation pass as waves of resident CTAs (0: two)
    bool sorted = false;
    int64_t s_n_opt = 0;
    int32_t *s_units = nullptr;
    double *s_values = nullptr;
    int64_t *s_off = nullptr;
    int32_t *s_jmap = nullptr;
    // Gamma term (esp_set_penalties): the loaded values, kept once penalties are first set
    double *values0 = nullptr;
    // the pass table tile by tile (units then values of each tile; one bulk copy per tile), when every
    // tile of the per-warp plan allows it; n_tiles: tiles of that plan
    unsigned char *il = nullptr;
    int64_t n_tiles = 0;
    bool il_f32 = false;             // il holds the units as fp32 bit patterns (every unit below 2^23)

    // factored placement table (esp_load_placement): no stored option table
    bool placement = false;
    DevPlace place = {};
    int32_t place_grid = 0;
    PlaceRes place_res = {};         // grid-resident placement solve (ESP_FLAG_RESIDENT), when allocated
    bool place_res_ok = false;
    bool hold_barrier = false;       // test hook: the next grid-resident solve's barrier never completes
    uint16_t *group = nullptr;
    int64_t *cap = nullptr;
    double *vmax = nullptr;
    int32_t *umax = nullptr;

    TileDesc *tiles = nullptr;
    int32_t *warp_begin = nullptr;
    bool il_enabled = true;          // later loads may interleave the pass table (esp_debug_set_interleave)
    bool il_f32_enabled = true;      // ... with fp32 units where exact (esp_debug_set_stage_f32)
    // failure-detection hooks (esp_debug.h): limit of a bounded wait of the evaluation passes in ms
    // (0: the default, 4 s), extra bytes announced on the next solve's first stage, allocations left
    // before an injected failure (-1: none)
    uint32_t wait_ms = 0;
    uint32_t hold_tx = 0;
    int64_t fail_alloc_in = -1;
    int32_t *scen_warps = nullptr;   // warps owning tiles of each scenario
    int32_t *scen_tiles = nullptr;   // tiles of each scenario
    int32_t *item_order = nullptr;   // the plan's ranges by the scenario of their first tile
    unsigned int *arrive = nullptr;  // per-scenario arrivals of the round pass in flight
    unsigned int *ver = nullptr;     // per-scenario price versions of the persistent pass
    unsigned int *work = nullptr;    // work items the persistent pass has handed out
    // persistent pass (every round in one cooperative launch): CTAs of its launch, 0 when the loaded
    // table cannot take it; persist_auto: plain solves use it by default; persist_mode: -1 automatic,
    // 0 never, 1 wherever the table can take it (esp_debug_set_persistent)
    int32_t persist_grid = 0;
    bool persist_auto = false;
    int persist_mode = -1;
    int32_t n_warps = 0, tile_opt = 0, grid = 0, uniform_k = 0;

    // cluster-resident kernel (tables without a group column): every cluster size that fits
    struct ResOption {
        ResPlan plan = {};
        int64_t smem = 0;
        int64_t n_max = 0;      // most options in one CTA's slice
        int32_t clusters = 0;   // clusters the device holds at once
    };
    std::vector<ResOption> res;
    int32_t *res_cuts = nullptr;
    int res_auto = -1;     // index into res of the automatic choice (-1: none fits)
    bool res_slower = false;   // the automatic choice is predicted slower than streaming: streaming runs
    int res_force = -1;    // index forced through esp_debug_resident (-1: automatic)

    double *lam = nullptr, *p64 = nullptr, *job_val = nullptr, *job_min = nullptr;
    double *best_dual = nullptr, *primal = nullptr, *dual = nullptr, *lambda0 = nullptr;
    float *p32 = nullptr, *ebound = nullptr;
    unsigned long long *U = nullptr, *U_final = nullptr, *hash = nullptr;
    int32_t *sel = nullptr, *rounds_run = nullptr, *converged = nullptr, *status = nullptr, *frozen = nullptr,
            *feasible = nullptr;
    unsigned int *err = nullptr;
    unsigned int *valflags = nullptr;
    // [0] exact resolutions (since the last read), [1] marked duplicates, [2] nanoseconds and [3] number
    // of the persistent pass's waits for a scenario's prices that had to poll
    unsigned long long *stats = nullptr;

    // trace buffers (grown on demand, freed on destroy)
    DevArr<double> lt;
    DevArr<long long> dt;
    DevArr<unsigned long long> ht;
    DevArr<double> gt;
    DevArr<unsigned long long> tt;

    cudaGraphExec_t gexec = nullptr;
    GraphKey gkey;
    // an event pair around the last solve or evaluation (esp_result::device_ms)
    cudaEvent_t solve_ev[2] = {nullptr, nullptr};
    // the stream of the table loads (the device's greatest priority) and the events that join it to
    // the context's stream (created by the first load)
    cudaStream_t load_stream = nullptr;
    cudaEvent_t load_ev[2] = {nullptr, nullptr};
    // profile of the last load (esp_debug_load_profile): host milliseconds of its phases, and the
    // cudaMalloc and cudaFree calls it made
    double load_ms[7] = {0, 0, 0, 0, 0, 0, 0};
    int64_t load_mallocs = 0, load_frees = 0;
    // pinned host staging of a load's validation result (its copy then does not block the host, which
    // plans the pass while the upload runs)
    unsigned char *h_stage = nullptr;
    size_t h_stage_bytes = 0;
    bool solve_timed = false;
    int64_t last_launches = 0;
    int32_t last_T = 0;

    // ESP_FLAG_PASS_EVENTS: event pairs around evaluation passes. Direct launches use ev_pool
    // (reused after a reset); a captured graph records into graph_pool, and every replay rewrites
    // those events, so they always hold the passes of the graph's latest replay.
    std::vector<cudaEvent_t> ev_pool;
    size_t ev_used = 0;
    std::vector<cudaEvent_t> graph_pool;
    size_t graph_pairs = 0;        // event pairs inside the cached graph
    bool graph_timed_run = false;  // a timed graph ran since the last reset
};

namespace {

esp_status cuda_fail(esp_ctx *c, cudaError_t e)
{
    (void)e;
    if (c)
        c->poisoned = true;
    return ESP_ERR_CUDA;
}

#define ESP_CUDA(call)                                  \
    do {                                                \
        cudaError_t e_ = (call);                        \
        if (e_ != cudaSuccess) {                        \
            cudaGetLastError();                         \
            return cuda_fail(ctx, e_);                  \
        }                                               \
    } while (0)

template <typename T>
esp_status dev_alloc(esp_ctx *ctx, T **p, size_t count, size_t pad_bytes = 64, bool zero = true)
{
    void *q = nullptr;
    const size_t bytes = count * sizeof(T) + pad_bytes;
    // reuse the smallest pooled buffer that fits and is at most about twice the size (a reload of a
    // table of the same shape gets every buffer back, without cudaMalloc / cudaFree; work still
    // queued on the context's stream that used it is ordered before the new contents)
    size_t best = SIZE_MAX, bi = SIZE_MAX;
    for (size_t i = 0; i < ctx->pool.size(); ++i) {
        const size_t have = ctx->pool[i].second;
        if (have >= bytes && have <= 2 * bytes + 4096 && have < best) {
            best = have;
            bi = i;
        }
    }
    size_t have = bytes;
    if (ctx->fail_alloc_in >= 0 && ctx->fail_alloc_in-- == 0)
        return ESP_ERR_OOM;   // injected failure (esp_debug_fail_alloc)
    if (bi != SIZE_MAX) {
        q = ctx->pool[bi].first;
        have = ctx->pool[bi].second;
        ctx->pool.erase(ctx->pool.begin() + (std::ptrdiff_t)bi);
    } else {
        ++ctx->load_mallocs;
        cudaError_t e = cudaMalloc(&q, bytes);
        if (e == cudaErrorMemoryAllocation) {
            cudaGetLastError();
            return ESP_ERR_OOM;
        }
        if (e != cudaSuccess)
            return cuda_fail(ctx, e);
    }
    ctx->table_bufs.emplace_back(q, have);
    if (zero) {   // buffers that a copy or kernel fills entirely skip this (zero = false)
        cudaError_t e = cudaMemsetAsync(q, 0, bytes, ctx->stream);
        if (e != cudaSuccess)
            return cuda_fail(ctx, e);
    }
    *p = static_cast<T *>(q);
    return ESP_OK;
}

// Frees the pooled buffers that the current table did not take.
void trim_pool(esp_ctx *ctx)
{
    for (auto &b : ctx->pool) {
        ++ctx->load_frees;
        cudaFree(b.first);
    }
    ctx->pool.clear();
}

// Drops the loaded table. keep = true (the start of a reload) moves its buffers to the pool, from which
// the next table's allocations are served; keep = false frees everything.
void release_table(esp_ctx *ctx, bool keep = false)
{
    // a reload keeps the executable graph: the next solve's key (which hashes every kernel argument)
    // decides whether it is replayed as it is, updated in place, or made anew
    if (ctx->gexec && !keep) {
        cudaGraphExecDestroy(ctx->gexec);
        ctx->gexec = nullptr;
        ctx->gkey = GraphKey();
    }
    if (keep) {
        ctx->pool.insert(ctx->pool.end(), ctx->table_bufs.begin(), ctx->table_bufs.end());
    } else {
        for (auto &b : ctx->table_bufs)
            cudaFree(b.first);
        trim_pool(ctx);
    }
    ctx->table_bufs.clear();
    ctx->res.clear();
    ctx->res_cuts = nullptr;
    ctx->sorted = false;
    ctx->s_n_opt = 0;
    ctx->s_units = nullptr;
    ctx->s_values = nullptr;
    ctx->s_off = nullptr;
    ctx->s_jmap = nullptr;
    ctx->values0 = nullptr;
    ctx->il = nullptr;
    ctx->il_f32 = false;
    ctx->persist_grid = 0;
    ctx->persist_auto = false;
    ctx->n_tiles = 0;
    ctx->placement = false;
    ctx->place = DevPlace{};
    ctx->place_grid = 0;
    ctx->place_res = PlaceRes{};
    ctx->place_res_ok = false;
    ctx->res_auto = -1;
    ctx->res_force = -1;
    ctx->loaded = false;
    ctx->solved = false;
}

template <typename T>
esp_status grow(esp_ctx *ctx, DevArr<T> &a, size_t n)
{
    if (a.n >= n && a.p)
        return ESP_OK;
    if (a.p)
        cudaFree(a.p);
    a.p = nullptr;
    a.n = 0;
    void *q = nullptr;
    cudaError_t e = cudaMalloc(&q, n * sizeof(T) + 64);
    if (e == cudaErrorMemoryAllocation) {
        cudaGetLastError();
        return ESP_ERR_OOM;
    }
    if (e != cudaSuccess)
        return cuda_fail(ctx, e);
    a.p = static_cast<T *>(q);
    a.n = n;
    return ESP_OK;
}

DevTable dev_table(const esp_ctx *c)
{
    DevTable t{};   // padding zeroed: the graph key hashes the kernel arguments byte by byte
    t.units = c->units;
    t.values = c->values;
    t.job_off = c->off;
    t.group = c->group;
    t.cap = c->cap;
    t.n_opt = c->n_opt;
    t.S = c->S;
    t.J = c->J;
    t.R = c->R;
    t.P = c->P;
    t.r_global = c->rg;
    t.n_groups = c->n_groups;
    t.small_units = c->small_units;
    t.jmap = nullptr;
    t.il = nullptr;
    t.il_f32 = 0;
    return t;
}

// The table the evaluation pass reads: the sorted layout when there is one, else the original.
DevTable pass_table(const esp_ctx *c)
{
    DevTable t = dev_table(c);
    if (c->sorted) {
        t.units = c->s_units;
        t.values = c->s_values;
        t.job_off = c->s_off;
        t.n_opt = c->s_n_opt;
        t.jmap = c->s_jmap;
    }
    t.il = c->il;
    t.il_f32 = (c->il != nullptr && c->il_f32) ? 1 : 0;
    return t;
}

DevState dev_state(const esp_ctx *c)
{
    DevState s{};
    s.lam = c->lam;
    s.p64 = c->p64;
    s.p32 = c->p32;
    s.ebound = c->ebound;
    s.U = c->U;
    s.U_final = c->U_final;
    s.hash = c->hash;
    s.sel = c->sel;
    s.job_val = c->job_val;
    s.job_min = c->job_min;
    s.rounds_run = c->rounds_run;
    s.converged = c->converged;
    s.status = c->status;
    s.frozen = c->frozen;
    s.best_dual = c->best_dual;
    s.primal = c->primal;
    s.dual = c->dual;
    s.feasible = c->feasible;
    s.vmax = c->vmax;
    s.umax = c->umax;
    s.err = c->err;
    s.stats = c->stats;
    s.arrive = c->arrive;
    s.ver = c->ver;
    s.work = c->work;
    s.lam_trace = nullptr;
    s.dem_trace = nullptr;
    s.hash_trace = nullptr;
    s.dual_trace = nullptr;
    s.time_trace = nullptr;
    return s;
}

esp_status check_ctx(esp_ctx *ctx)
{
    if (!ctx)
        return ESP_ERR_INVALID_ARG;
    if (ctx->poisoned)
        return ESP_ERR_STATE;
    return ESP_OK;
}

esp_status check_shape(int32_t S, int32_t J, int32_t R, int32_t P, int32_t rg, bool grouped, int32_t *n_groups)
{
    if (S < 1 || J < 0 || R < 1 || R > kMaxR || P < 1)
        return ESP_ERR_INVALID_ARG;
    if (!grouped) {
        if (P != R || rg != R)
            return ESP_ERR_INVALID_ARG;
        *n_groups = 0;
        return ESP_OK;
    }
    if (rg < 0 || rg >= R)
        return ESP_ERR_INVALID_ARG;
    const int32_t per = R - rg;
    if (P <= rg || (P - rg) % per != 0)
        return ESP_ERR_INVALID_ARG;
    const int32_t ng = (P - rg) / per;
    if (ng < 1 || ng > 65536)
        return ESP_ERR_INVALID_ARG;
    *n_groups = ng;
    return ESP_OK;
}

// Per-scenario and per-job state of a solve (prices, demands, selections, objectives, status).
esp_status alloc_solve_state(esp_ctx *ctx)
{
    const size_t S = (size_t)ctx->S, SP = (size_t)ctx->S * ctx->P, SJ = (size_t)ctx->S * ctx->J;
    esp_status a = ESP_OK;
    auto al = [&](auto **p, size_t n) {
        if (a == ESP_OK)
            a = dev_alloc(ctx, p, n);
    };
    al(&ctx->lam, SP);
    al(&ctx->p64, SP);
    al(&ctx->p32, SP);
    al(&ctx->ebound, S);
    al(&ctx->U, SP);
    al(&ctx->U_final, SP);
    al(&ctx->hash, S);
    al(&ctx->sel, SJ);
    al(&ctx->job_val, SJ);
    al(&ctx->job_min, SJ);
    al(&ctx->rounds_run, S);
    al(&ctx->converged, S);
    al(&ctx->status, S);
    al(&ctx->frozen, S);
    al(&ctx->feasible, S);
    al(&ctx->best_dual, S);
    al(&ctx->primal, S);
    al(&ctx->dual, S);
    al(&ctx->lambda0, SP);
    al(&ctx->ver, S);
    al(&ctx->work, 1);
    al(&ctx->err, 4);
    return a;
}

// A table load's device work (copies, validation, duplicate marks, sorted layout, interleaved tiles,
// solve state) runs on a stream of the context with the device's greatest priority, joined to the
// context's stream by an event on each side: it is ordered exactly as on the context's stream, and a
// load that overlaps another context's solve gets SMs as soon as the solve's passes free them
// instead of queueing behind them (measured on the heavy-tailed table: the 22 ms reload then hides
// under the other context's 320 ms solve).
class LoadStreamScope {
public:
    explicit LoadStreamScope(esp_ctx *c) : ctx_(c), user_(c->stream) {}
    LoadStreamScope(const LoadStreamScope &) = delete;
    LoadStreamScope &operator=(const LoadStreamScope &) = delete;

    esp_status begin()
    {
        if (cudaSetDevice(ctx_->device) != cudaSuccess)
            return cuda_fail(ctx_, cudaGetLastError());
        if (!ctx_->load_stream) {
            int lo = 0, hi = 0;
            cudaError_t e = cudaDeviceGetStreamPriorityRange(&lo, &hi);
            if (e == cudaSuccess)
                e = cudaStreamCreateWithPriority(&ctx_->load_stream, cudaStreamNonBlocking, hi);
            for (int i = 0; i < 2 && e == cudaSuccess; ++i)
                e = cudaEventCreateWithFlags(&ctx_->load_ev[i], cudaEventDisableTiming);
            if (e != cudaSuccess)
                return cuda_fail(ctx_, e);
        }
        cudaError_t e = cudaEventRecord(ctx_->load_ev[0], user_);
        if (e == cudaSuccess)
            e = cudaStreamWaitEvent(ctx_->load_stream, ctx_->load_ev[0], 0);
        if (e != cudaSuccess)
            return cuda_fail(ctx_, e);
        ctx_->stream = ctx_->load_stream;
        active_ = true;
        return ESP_OK;
    }
    ~LoadStreamScope()
    {
        if (!active_)
            return;
        // later work on the context's stream (solves) is ordered after everything the load queued
        if (cudaEventRecord(ctx_->load_ev[1], ctx_->load_stream) != cudaSuccess ||
            cudaStreamWaitEvent(user_, ctx_->load_ev[1], 0) != cudaSuccess) {
            cudaGetLastError();
            cudaStreamSynchronize(ctx_->load_stream);
        }
        ctx_->stream = user_;
    }

private:
    esp_ctx *ctx_;
    cudaStream_t user_;
    bool active_ = false;
};

// Upload (host or device source), validate on the device, plan, allocate the solve state.
esp_status load_common(esp_ctx *ctx, int32_t S, int32_t J, int32_t R, int32_t P, int32_t rg, const int64_t *job_off,
                       const int32_t *units, const double *values, const uint16_t *group, const int64_t *capacity,
                       bool device_src)
{
    esp_status st = check_ctx(ctx);
    if (st != ESP_OK)
        return st;
    if (!job_off || !capacity || (J > 0 && (!units || !values)))
        return ESP_ERR_INVALID_ARG;
    int32_t n_groups = 0;
    const bool grouped = group != nullptr;
    if ((st = check_shape(S, J, R, P, rg, grouped, &n_groups)) != ESP_OK)
        return st;
    if (!grouped)
        rg = R;
    ESP_CUDA(cudaSetDevice(ctx->device));
    const auto t_start = std::chrono::steady_clock::now();
    auto since = [&]() {
        return std::chrono::duration<double, std::milli>(std::chrono::steady_clock::now() - t_start).count();
    };
    ctx->load_mallocs = ctx->load_frees = 0;
    for (double &x : ctx->load_ms)
        x = 0.0;
    release_table(ctx, true);

    const int64_t n_jobs = (int64_t)S * J;
    std::vector<int64_t> h_off;
    const int64_t *off_host = job_off;
    if (device_src) {
        h_off.resize(n_jobs + 1);
        ESP_CUDA(cudaMemcpyAsync(h_off.data(), job_off, (n_jobs + 1) * sizeof(int64_t), cudaMemcpyDeviceToHost,
                                 ctx->stream));
        ESP_CUDA(cudaStreamSynchronize(ctx->stream));
        off_host = h_off.data();
    }
    const int64_t n_opt = off_host[n_jobs];
    if (off_host[0] != 0 || n_opt < n_jobs || n_opt > ((int64_t)1 << 40))
        return ESP_ERR_INVALID_ARG;

    ctx->S = S;
    ctx->J = J;
    ctx->R = R;
    ctx->P = P;
    ctx->rg = rg;
    ctx->n_groups = n_groups;
    ctx->n_opt = n_opt;

#define ALLOC(ptr, count)                                 \
    do {                                                  \
        esp_status a_ = dev_alloc(ctx, &(ptr), (count));  \
        if (a_ != ESP_OK) {                               \
            release_table(ctx);                           \
            return a_;                                    \
        }                                                 \
    } while (0)
// a buffer that a copy or a kernel of this load fills entirely (not zeroed first)
#define ALLOC_FILLED(ptr, count)                                         \
    do {                                                                 \
        esp_status a_ = dev_alloc(ctx, &(ptr), (count), 64, false);      \
        if (a_ != ESP_OK) {                                              \
            release_table(ctx);                                          \
            return a_;                                                   \
        }                                                                \
    } while (0)

    ALLOC_FILLED(ctx->units, (size_t)n_opt * R);
    ALLOC_FILLED(ctx->values, (size_t)n_opt);
    ALLOC_FILLED(ctx->off, (size_t)n_jobs + 1);
    ctx->group = nullptr;
    if (grouped)
        ALLOC_FILLED(ctx->group, (size_t)n_opt);
    ALLOC_FILLED(ctx->cap, (size_t)S * P);
    ALLOC(ctx->vmax, (size_t)S);
    ALLOC(ctx->umax, (size_t)S * R);
    ALLOC(ctx->valflags, 4);
    ALLOC(ctx->stats, 4);

    const cudaMemcpyKind kind = device_src ? cudaMemcpyDeviceToDevice : cudaMemcpyHostToDevice;
    ESP_CUDA(cudaMemcpyAsync(ctx->units, units, (size_t)n_opt * R * sizeof(int32_t), kind, ctx->stream));
    ESP_CUDA(cudaMemcpyAsync(ctx->values, values, (size_t)n_opt * sizeof(double), kind, ctx->stream));
    ESP_CUDA(cudaMemcpyAsync(ctx->off, job_off, (size_t)(n_jobs + 1) * sizeof(int64_t), kind, ctx->stream));
    if (grouped)
        ESP_CUDA(cudaMemcpyAsync(ctx->group, group, (size_t)n_opt * sizeof(uint16_t), kind, ctx->stream));
    ESP_CUDA(cudaMemcpyAsync(ctx->cap, capacity, (size_t)S * P * sizeof(int64_t), kind, ctx->stream));

    // validation, then (stream-ordered after it) the marking of duplicates in the device copy; the
    // host plans the pass meanwhile, and checks the validation result before anything uses the plan
    const DevTable t = dev_table(ctx);
    ESP_CUDA(launch_validate(t, ctx->vmax, ctx->umax, ctx->valflags, ctx->stream));
    const size_t stage_bytes = 16 + (size_t)S * R * sizeof(int32_t);
    if (ctx->h_stage_bytes < stage_bytes) {
        if (ctx->h_stage)
            cudaFreeHost(ctx->h_stage);
        ctx->h_stage = nullptr;
        ctx->h_stage_bytes = 0;
        void *hp = nullptr;
        if (cudaHostAlloc(&hp, stage_bytes, cudaHostAllocDefault) != cudaSuccess) {
            cudaGetLastError();
            cudaStreamSynchronize(ctx->stream);
            release_table(ctx);
            return ESP_ERR_OOM;
        }
        ctx->h_stage = static_cast<unsigned char *>(hp);
        ctx->h_stage_bytes = stage_bytes;
    }
    unsigned int *h_vflags = reinterpret_cast<unsigned int *>(ctx->h_stage);
    const int32_t *h_umax = reinterpret_cast<const int32_t *>(ctx->h_stage + 16);
    ESP_CUDA(cudaMemcpyAsync(h_vflags, ctx->valflags, sizeof(unsigned int), cudaMemcpyDeviceToHost, ctx->stream));
    ESP_CUDA(cudaMemcpyAsync(ctx->h_stage + 16, ctx->umax, (size_t)S * R * sizeof(int32_t), cudaMemcpyDeviceToHost,
                             ctx->stream));
    ctx->load_ms[0] = since();   // uploads and validation queued
    // the plan of the previous load serves when the shape and offsets are the same
    PlanCache &pc = ctx->pc;
    const bool cached = pc.valid && pc.S == S && pc.J == J && pc.R == R && pc.P == P && pc.grouped == grouped &&
                        pc.sorted_enabled == ctx->sorted_enabled && (int64_t)pc.off.size() == n_jobs + 1 &&
                        std::memcmp(pc.off.data(), off_host, (size_t)(n_jobs + 1) * sizeof(int64_t)) == 0;
    // option counts, on the host meanwhile: every job non-empty makes the offsets strictly
    // increasing up to n_opt, so no kernel below can index outside the table
    int64_t max_k = 1, min_k = n_jobs ? INT64_MAX : 1;
    if (cached) {
        max_k = pc.max_k;
        min_k = pc.min_k;
    } else {
        for (int64_t j = 0; j < n_jobs; ++j) {
            const int64_t k = off_host[j + 1] - off_host[j];
            max_k = std::max<int64_t>(max_k, k);
            min_k = std::min<int64_t>(min_k, k);
        }
    }
    if (min_k < 1) {
        cudaStreamSynchronize(ctx->stream);
        release_table(ctx);
        return ESP_ERR_INVALID_ARG;
    }
    ctx->max_k = max_k;
    ESP_CUDA(launch_mark_duplicates(t, ctx->units, ctx->stats + 1, ctx->stream, max_k));

    // plan the evaluation pass
    ctx->uniform_k = (!grouped && min_k == max_k && max_k <= 32 && (max_k & (max_k - 1)) == 0) ? (int32_t)max_k : 0;

    // general tables without a group column: the evaluation pass reads the sorted layout (runs of
    // equal-size jobs take the uniform paths). Jobs keep their option order, so the copy inherits
    // the duplicate marks of the original; its padding is marked as it is written.
    SortedLayout lay_new;
    bool use_sorted = false;
    if (cached)
        use_sorted = pc.sorted;
    else
        use_sorted = ctx->sorted_enabled && !grouped && ctx->uniform_k == 0 && J >= 1 &&
                     sort_layout(off_host, S, J, lay_new, kRunMaxK);
    const SortedLayout &lay = cached ? pc.lay : lay_new;
    if (use_sorted) {
        const int64_t sn = lay.off.back();
        ALLOC_FILLED(ctx->s_units, (size_t)sn * R);   // every option of the layout, padding included
        ALLOC_FILLED(ctx->s_values, (size_t)sn);
        ALLOC_FILLED(ctx->s_off, (size_t)n_jobs + 1);
        ALLOC_FILLED(ctx->s_jmap, (size_t)n_jobs);
        ESP_CUDA(cudaMemcpyAsync(ctx->s_off, lay.off.data(), lay.off.size() * sizeof(int64_t), cudaMemcpyHostToDevice,
                                 ctx->stream));
        ESP_CUDA(cudaMemcpyAsync(ctx->s_jmap, lay.jmap.data(), lay.jmap.size() * sizeof(int32_t),
                                 cudaMemcpyHostToDevice, ctx->stream));
        ctx->s_n_opt = sn;
        ctx->sorted = true;
        ESP_CUDA(launch_gather_sorted(dev_table(ctx), pass_table(ctx), ctx->s_units, ctx->s_values, ctx->stream));
    }
    ctx->load_ms[1] = since();   // sorted layout queued
    const int64_t *plan_off = ctx->sorted ? lay.off.data() : off_host;
    const int32_t *plan_scen = ctx->sorted ? lay.scen.data() : nullptr;
    const int32_t *plan_runk = ctx->sorted ? lay.runk.data() : nullptr;

    Plan plan_new;
    const int tile_opt = tile_options_for(R, grouped, max_k, ctx->uniform_k >= 4);
    // a sorted layout's tiles are runs and chunks only (the sorted layout exists only without a group
    // column): the runs-only instantiation
    const int mode = ctx->uniform_k > 0 ? kModeUniform : (use_sorted && !grouped) ? kModeRuns : kModeGeneral;
    int per_sm = pass_ctas_per_sm(R, grouped, mode, P, tile_opt);
    // a table that may take the persistent pass is planned for its co-resident CTAs, so that each of
    // its physical warps runs exactly `waves` ranges (its fp32 stage units are decided after the
    // validation; a table that turns out not to qualify runs the same plan with per-round launches)
    const int per_sm_persist = (ctx->il_enabled && ctx->il_f32_enabled && pass_f32_shape(R, grouped, mode))
                                   ? pass_persist_ctas_per_sm(R, mode, P, tile_opt)
                                   : 0;
    if (per_sm_persist > 0 && per_sm_persist < per_sm)
        per_sm = per_sm_persist;
    ctx->load_ms[2] = since();   // occupancy of the pass kernels
    if (per_sm < 1) {
        cudaStreamSynchronize(ctx->stream);
        release_table(ctx);
        return ESP_ERR_UNSUPPORTED;
    }
    // Ranges of the plan as waves of resident CTAs: two by default (with per-round launches, CTAs that
    // finish early take the second wave's ranges; the persistent pass hands them out as work items,
    // two per warp and round), one for a sorted layout (measured 2% faster there).
    const int waves = ctx->plan_waves > 0 ? ctx->plan_waves : (mode == kModeRuns) ? 1 : 2;
    const int max_warps = ctx->sm_count * per_sm * kWarpsPerCta * waves;
    const bool plan_cached = cached && pc.max_warps == max_warps && pc.tile_opt == tile_opt;
    if (!plan_cached && (!plan_tiles(plan_off, S, J, tile_opt, max_warps, plan_new, plan_scen, plan_runk) ||
                         !check_plan(plan_off, S, J, plan_new, plan_scen, plan_runk))) {
        cudaStreamSynchronize(ctx->stream);
        release_table(ctx);
        return ESP_ERR_INVALID_ARG;
    }
    const Plan &plan = plan_cached ? pc.plan : plan_new;
    // the runs-only instantiation has no path for a general tile
    if (mode == kModeRuns)
        for (const TileDesc &d : plan.tiles)
            if (!(d.flags & (TILE_RUN | TILE_BIG))) {
                cudaStreamSynchronize(ctx->stream);
                release_table(ctx);
                return ESP_ERR_INVALID_ARG;
            }
    // the validation result (the copies, validation and duplicate marking ran during the planning)
    ctx->load_ms[3] = since();   // planned
    ESP_CUDA(cudaStreamSynchronize(ctx->stream));
    ctx->load_ms[4] = since();   // uploads, validation and marks done
    const unsigned int vflags = *h_vflags;
    if (vflags != 0) {
        release_table(ctx);
        return ESP_ERR_INVALID_ARG;
    }
    ctx->small_units = 1;
    for (size_t i = 0; i < (size_t)S * R; ++i)
        if (h_umax[i] >= (1 << 23))
            ctx->small_units = 0;
    ALLOC(ctx->scen_warps, (size_t)S);
    ALLOC(ctx->scen_tiles, (size_t)S);
    ALLOC(ctx->item_order, (size_t)std::max<int32_t>(plan.n_warps, 1));
    ALLOC(ctx->arrive, (size_t)S);
    {
        ctx->n_warps = plan.n_warps;
        ctx->tile_opt = plan.tile_opt;
        ctx->grid = (plan.n_warps + kWarpsPerCta - 1) / kWarpsPerCta;
        ALLOC(ctx->tiles, plan.tiles.size() + 1);
        ALLOC(ctx->warp_begin, plan.warp_begin.size());
        std::vector<int32_t> sw((size_t)S, 0);
        for (int32_t w = 0; w < plan.n_warps; ++w) {
            int32_t last = -1;
            for (int32_t k = plan.warp_begin[w]; k < plan.warp_begin[w + 1]; ++k)
                if (plan.tiles[k].scenario != last) {
                    last = plan.tiles[k].scenario;
                    ++sw[last];
                }
        }
        std::vector<int32_t> stl((size_t)S, 0);
        for (const TileDesc &d : plan.tiles)
            ++stl[d.scenario];
        ESP_CUDA(cudaMemcpyAsync(ctx->scen_warps, sw.data(), sw.size() * sizeof(int32_t), cudaMemcpyHostToDevice,
                                 ctx->stream));
        ESP_CUDA(cudaMemcpyAsync(ctx->scen_tiles, stl.data(), stl.size() * sizeof(int32_t), cudaMemcpyHostToDevice,
                                 ctx->stream));
        // the ranges by the scenario of their first tile, in table order within a scenario (a sorted
        // layout keeps each scenario's runs, large jobs and one- and two-option jobs apart)
        std::vector<int32_t> order((size_t)plan.n_warps);
        for (int32_t w = 0; w < plan.n_warps; ++w)
            order[w] = w;
        auto first_scen = [&](int32_t w) {
            const int32_t k = plan.warp_begin[w];
            return k < (int32_t)plan.tiles.size() ? plan.tiles[k].scenario : S;
        };
        std::stable_sort(order.begin(), order.end(),
                         [&](int32_t x, int32_t y) { return first_scen(x) < first_scen(y); });
        if (!order.empty())
            ESP_CUDA(cudaMemcpyAsync(ctx->item_order, order.data(), order.size() * sizeof(int32_t),
                                     cudaMemcpyHostToDevice, ctx->stream));
        ESP_CUDA(cudaStreamSynchronize(ctx->stream));
        if (!plan.tiles.empty())
            ESP_CUDA(cudaMemcpyAsync(ctx->tiles, plan.tiles.data(), plan.tiles.size() * sizeof(TileDesc),
                                     cudaMemcpyHostToDevice, ctx->stream));
        ESP_CUDA(cudaMemcpyAsync(ctx->warp_begin, plan.warp_begin.data(), plan.warp_begin.size() * sizeof(int32_t),
                                 cudaMemcpyHostToDevice, ctx->stream));
        // one bulk copy per tile when every tile can take it: no job offsets needed (uniform tables,
        // runs and chunks of the sorted layout), every tile 16-byte aligned in the interleaved copy,
        // and its values aligned in the stage for the loads of its path (16 bytes for the paths of
        // four options per lane, 8 otherwise)
        const int64_t W = 4 * (int64_t)R + 8;
        bool il_ok = ctx->il_enabled && !grouped && (ctx->uniform_k > 0 || ctx->sorted) && !plan.tiles.empty();
        for (size_t k = 0; il_ok && k < plan.tiles.size(); ++k) {
            const TileDesc &d = plan.tiles[k];
            const int kk = (d.flags & TILE_RUN) ? tile_run_k(d.flags) : ctx->uniform_k;
            const bool vec = (d.flags & TILE_BIG) ? ((d.opt_begin | (int64_t)d.n_opt) & 3) == 0 : kk >= 4;
            il_ok = (d.opt_begin * W) % 16 == 0 && ((int64_t)d.n_opt * R * 4) % (vec ? 16 : 8) == 0 &&
                    ((d.flags & (TILE_BIG | TILE_RUN)) || ctx->uniform_k > 0);
        }
        if (il_ok) {
            const int64_t pass_opt = ctx->sorted ? ctx->s_n_opt : n_opt;
            ALLOC_FILLED(ctx->il, (size_t)(pass_opt * W));   // the tiles cover every option
            ctx->n_tiles = (int64_t)plan.tiles.size();
            // units as fp32 where every unit converts exactly and the shape has that instantiation
            ctx->il_f32 = ctx->il_f32_enabled && ctx->small_units && pass_f32_shape(R, grouped, mode);
            ESP_CUDA(launch_interleave(pass_table(ctx), ctx->tiles, ctx->n_tiles, ctx->il, ctx->il_f32,
                                       ctx->stream));
            // the persistent pass: every CTA of its launch co-resident, no more warps than ranges. Used
            // by default on uniform tables with at least kPersistMinTiles tiles per warp of its launch
            // (measured on the what-if batch at 1024 and 256 scenarios: 16% and 19% faster per solve;
            // at 64 scenarios, 4.5 tiles per warp, 5% slower; sorted layouts measured faster with
            // per-round launches)
            if (ctx->il_f32 && per_sm_persist > 0 && plan.n_warps > 0) {
                const int64_t cap_ctas = (int64_t)per_sm_persist * ctx->sm_count;
                const int64_t need_ctas = ((int64_t)plan.n_warps + kWarpsPerCta - 1) / kWarpsPerCta;
                ctx->persist_grid = (int32_t)std::min(cap_ctas, need_ctas);
                ctx->persist_auto = mode == kModeUniform &&
                                    ctx->n_tiles >= (int64_t)kPersistMinTiles * ctx->persist_grid * kWarpsPerCta;
            }
        }
    }

    // the resident kernel's options are planned on first use (plan_resident_options)
    ctx->res_planned = false;

#undef ALLOC
#undef ALLOC_FILLED
    if ((st = alloc_solve_state(ctx)) != ESP_OK) {
        release_table(ctx);
        return st;
    }
    ESP_CUDA(cudaStreamSynchronize(ctx->stream));
    if (!plan_cached) {   // keep this load's plan for the next load of the same offsets
        pc.valid = true;
        pc.S = S;
        pc.J = J;
        pc.R = R;
        pc.P = P;
        pc.grouped = grouped;
        pc.sorted_enabled = ctx->sorted_enabled;
        if (!cached) {
            pc.off.assign(off_host, off_host + n_jobs + 1);
            pc.min_k = min_k;
            pc.max_k = max_k;
            pc.sorted = use_sorted;
            pc.lay = std::move(lay_new);
        }
        pc.max_warps = max_warps;
        pc.tile_opt = tile_opt;
        pc.plan = std::move(plan_new);
    }
    ctx->load_ms[5] = since();   // tiles, interleaved table and solve state queued
    trim_pool(ctx);
    ctx->load_ms[6] = since();
    ctx->loaded = true;
    ctx->solved = false;
    return ESP_OK;
}

esp_status check_params(const esp_ctx *ctx, const esp_params *p)
{
    if (!p)
        return ESP_ERR_INVALID_ARG;
    if (!(p->eta0 > 0.0) || !std::isfinite(p->eta0))
        return ESP_ERR_INVALID_ARG;
    if (p->step != ESP_STEP_FIXED && p->step != ESP_STEP_INV_SQRT)
        return ESP_ERR_INVALID_ARG;
    if (p->mode != ESP_PRICE_RAW && p->mode != ESP_PRICE_NORMALIZED)
        return ESP_ERR_INVALID_ARG;
    if (p->max_rounds < 0 || p->max_rounds > 100000000)
        return ESP_ERR_INVALID_ARG;
    if (!(p->tol >= 0.0) || !std::isfinite(p->tol))
        return ESP_ERR_INVALID_ARG;
    if (p->flags & ~(uint32_t)(ESP_FLAG_EXACT_ONLY | ESP_FLAG_PER_ROUND_LAUNCH | ESP_FLAG_PASS_EVENTS | ESP_FLAG_RESIDENT))
        return ESP_ERR_INVALID_ARG;
    if (p->lambda0) {
        const size_t n = (size_t)ctx->S * ctx->P;
        for (size_t i = 0; i < n; ++i)
            if (!(p->lambda0[i] >= 0.0) || !std::isfinite(p->lambda0[i]))
                return ESP_ERR_INVALID_ARG;
    }
    return ESP_OK;
}

// Every device buffer the solve kernels touch exists (an internal inconsistency is reported on the
// host instead of reaching a kernel as a null pointer).
bool state_ready(const esp_ctx *c)
{
    const void *need[] = {c->lam, c->p64, c->p32, c->ebound, c->U, c->U_final, c->hash, c->sel, c->job_val,
                          c->job_min, c->rounds_run, c->converged, c->status, c->frozen, c->feasible,
                          c->best_dual, c->primal, c->dual, c->lambda0, c->err, c->vmax, c->umax, c->stats,
                          c->arrive, c->ver, c->work, c->cap, c->scen_warps};
    for (const void *p : need)
        if (!p)
            return false;
    if (c->placement)
        return c->place.cfg_units && c->place.cfg_values && c->place.sens && c->place.job_type &&
               c->place.node_type && c->place.D && c->place.cfg_dup && c->place.warp_job && c->place.n_warps > 0;
    return c->grid == 0 || (c->tiles && c->warp_begin && c->units && c->values && c->off);
}

// The plan of the evaluation pass as the kernels take it.
DevPlan dev_plan(const esp_ctx *c, bool fused)
{
    DevPlan pl{};
    pl.tiles = c->tiles;
    pl.warp_begin = c->warp_begin;
    pl.n_warps = c->n_warps;
    pl.tile_opt = c->tile_opt;
    pl.uniform_k = c->uniform_k;
    pl.runs_only = (c->sorted && c->group == nullptr) ? 1 : 0;
    pl.scen_warps = fused ? c->scen_warps : nullptr;
    pl.scen_tiles = c->scen_tiles;
    pl.item_order = c->item_order;
    return pl;
}

// Solve arguments common to every launch of a solve or evaluation.
SolveArgs solve_args(const esp_ctx *c, double eta0, int32_t step, int32_t mode, int32_t T, double tol, uint32_t flags)
{
    SolveArgs a{};
    a.eta0 = eta0;
    a.step = step;
    a.mode = mode;
    a.T = T;
    a.tol = tol;
    a.flags = flags;
    a.exact_only = (flags & ESP_FLAG_EXACT_ONLY) ? 1 : 0;
    a.wait_ms = c->wait_ms ? c->wait_ms : kWaitLimitMs;
    a.hold_tx = c->hold_tx;
    return a;
}

// Options of the cluster-resident kernel (ESP_FLAG_RESIDENT) for the loaded table: every cluster
// size whose slices fit one CTA's shared memory, with the automatic choice. Planned on first use
// (not every load needs them), from the host copy of the offsets kept with the plan.
esp_status plan_resident_options(esp_ctx *ctx)
{
    if (ctx->res_planned)
        return ESP_OK;
    ctx->res_planned = true;
    ctx->res.clear();
    ctx->res_auto = -1;
    ctx->res_slower = false;
    const int32_t S = ctx->S, J = ctx->J, R = ctx->R;
    esp_status st = ESP_OK;
    if (!ctx->pc.valid || (int64_t)ctx->pc.off.size() != (int64_t)S * J + 1)
        return ESP_OK;
    if (ctx->group == nullptr && J >= 1) {
        int optin = 0;
        ESP_CUDA(cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, ctx->device));
        const int32_t rk = (ctx->pc.min_k == ctx->pc.max_k) ? (int32_t)ctx->pc.max_k : 0;
        std::vector<ResShape> shapes;
        for (int32_t cs = 1; cs <= kResMaxCluster; cs *= 2) {
            ResShape sh;
            if (!plan_resident(ctx->pc.off.data(), S, J, cs, sh) || sh.n_max > (1 << 24))
                continue;
            esp_ctx::ResOption o;
            o.plan.cs = cs;
            o.plan.k = rk;
            o.plan.m_pad = (sh.m_max + 31) & ~31;
            o.plan.n_cap = (sh.n_max + 1) & ~1LL;
            o.smem = res_smem_bytes(R, o.plan);
            o.n_max = sh.n_max;
            if (o.smem > optin)
                continue;
            int nc = 0;
            ESP_CUDA(res_max_clusters(dev_table(ctx), o.plan, ctx->small_units != 0, &nc));
            if (nc < 1)
                continue;
            o.clusters = nc;
            ctx->res.push_back(o);
            shapes.push_back(std::move(sh));
        }
        if (!ctx->res.empty()) {
            size_t total = 0;
            for (const ResShape &sh : shapes)
                total += sh.cuts.size();
            if ((st = dev_alloc(ctx, &ctx->res_cuts, total)) != ESP_OK) {
                ctx->res.clear();            // no option without its slices; a later solve plans again
                ctx->res_planned = false;
                return st;
            }
            size_t at = 0;
            for (size_t i = 0; i < shapes.size(); ++i) {
                ESP_CUDA(cudaMemcpyAsync(ctx->res_cuts + at, shapes[i].cuts.data(), shapes[i].cuts.size() * sizeof(int32_t),
                                         cudaMemcpyHostToDevice, ctx->stream));
                ctx->res[i].plan.cuts = ctx->res_cuts + at;
                at += shapes[i].cuts.size();
            }
            ESP_CUDA(cudaStreamSynchronize(ctx->stream));
            // automatic size: most scenario-rounds per microsecond under a simple cost model, a fixed
            // cost per round (barriers and the price update; smaller without a cluster) plus the
            // slice's options at the SM's screening rate; ties keep the smaller cluster
            double best = -1.0;
            for (size_t i = 0; i < ctx->res.size(); ++i) {
                const esp_ctx::ResOption &o = ctx->res[i];
                const double round_us = (o.plan.cs == 1 ? 0.6 : 1.0) + 7.8e-5 * (double)o.n_max;
                const double rate = (double)std::min<int64_t>(S, o.clusters) / round_us;
                if (rate > best * 1.02) {
                    best = rate;
                    ctx->res_auto = (int)i;
                }
            }
            // the automatic choice runs only where it is predicted faster than streaming. Absolute
            // times per round measured on GB300: a resident round of one wave of clusters costs about
            // 2.6 + 0.135 cs + 7.8e-5 n_max us (2.7 us at 1 CTA, 4.75 us at 16 CTAs), and S scenarios
            // take ceil(S / clusters) waves; a streaming round reads the table at about 5.6 TB/s
            // plus 3 us, and no streaming round takes less than about 9 us (launch and update latency)
            if (ctx->res_auto >= 0) {
                const esp_ctx::ResOption &o = ctx->res[ctx->res_auto];
                const double waves = std::ceil((double)S / (double)o.clusters);
                const double res_us = waves * (2.6 + 0.135 * o.plan.cs + 7.8e-5 * (double)o.n_max);
                const double bytes = (double)ctx->n_opt * (4.0 * R + 8.0);
                const double stream_us = std::max(9.0, 3.0 + bytes / 5.6e6);
                ctx->res_slower = res_us > stream_us;
            }
        }
    }

    return ESP_OK;
}

// Whether the passes of this table are launched as programmatic dependents by default: measured
// on GB300 it pays for large uniform tables (what-if batch: -1.2% per solve) and costs on others
// (one 2048-job scenario: +10%; the ragged 16-scenario table: +12%), so only the former use it.
bool pdl_default(const esp_ctx *c)
{
    return !c->placement && c->uniform_k > 0 && (int64_t)c->S * c->J >= (1 << 16);
}

// Records event i of the pair around a solve on the context's stream (outside any capture).
cudaError_t record_solve_event(esp_ctx *ctx, int i)
{
    if (!ctx->solve_ev[i]) {
        const cudaError_t e = cudaEventCreate(&ctx->solve_ev[i]);
        if (e != cudaSuccess)
            return e;
    }
    ctx->solve_timed = (i == 1);
    return cudaEventRecord(ctx->solve_ev[i], ctx->stream);
}

// Queues one whole solve on the stream (captured into a graph when the stream allows it).
esp_status enqueue_solve(esp_ctx *ctx, const esp_params *p, const DevState &st, bool has_l0)
{
    if (!state_ready(ctx))
        return ESP_ERR_STATE;
    const DevTable t = pass_table(ctx);
    const DevTable t_orig = dev_table(ctx);   // the resident kernel reads the original layout
    // the last warp to finish a scenario in a round pass updates its prices (one launch per round);
    // ESP_FLAG_PER_ROUND_LAUNCH keeps a separate update launch (also used when no warp has tiles)
    const bool fused = ctx->grid > 0 && !(p->flags & ESP_FLAG_PER_ROUND_LAUNCH);
    const DevPlan pl = dev_plan(ctx, fused);
    const SolveArgs a = solve_args(ctx, p->eta0, p->step, p->mode, p->max_rounds, p->tol, p->flags);
    ctx->hold_tx = 0;   // the hook holds one solve only
    const int T = p->max_rounds;

    const bool timed = (p->flags & ESP_FLAG_PASS_EVENTS) != 0;
    const bool use_graph = ctx->stream != nullptr;   // the legacy default stream cannot be captured
    std::vector<cudaEvent_t> &pool = use_graph ? ctx->graph_pool : ctx->ev_pool;
    size_t pool_used = use_graph ? 0 : ctx->ev_used;
    if ((p->flags & ESP_FLAG_RESIDENT) && !ctx->placement) {
        const esp_status rs = plan_resident_options(ctx);
        if (rs != ESP_OK)
            return rs;
    }
    const int ri = (p->flags & ESP_FLAG_RESIDENT) && !ctx->placement
                       ? (ctx->res_force >= 0 ? ctx->res_force : (ctx->res_slower ? -1 : ctx->res_auto))
                       : -1;
    // a placement table solves all rounds in one cooperative launch when asked, unless the
    // fingerprint or dual trace is wanted (those need the per-round launches)
    const bool place_res = ctx->placement && (p->flags & ESP_FLAG_RESIDENT) && ctx->place_res_ok &&
                           st.hash_trace == nullptr && st.dual_trace == nullptr;
    const bool hold = place_res && ctx->hold_barrier;
    ctx->hold_barrier = false;
    // rounds 0 .. T-1 in one persistent launch (fused updates, fp32 stage units, no per-pass events,
    // no fingerprint or dual trace: those are written by the round passes)
    const bool persist = ctx->persist_grid > 0 && (ctx->persist_mode > 0 || (ctx->persist_mode < 0 && ctx->persist_auto)) &&
                         !ctx->placement && ri < 0 && fused &&
                         !timed && t.il_f32 && T > 0 && st.hash_trace == nullptr && st.dual_trace == nullptr &&
                         (int64_t)T * ctx->n_tiles < (int64_t)INT32_MAX;   // items and a warp's tiles below 2^31
    auto timed_launch = [&](auto &&launch) -> cudaError_t {
        if (!timed)
            return launch();
        while (pool.size() < pool_used + 2) {
            cudaEvent_t ev;
            cudaError_t e = cudaEventCreate(&ev);
            if (e != cudaSuccess)
                return e;
            pool.push_back(ev);
        }
        // external records: inside a stream capture they become event-record nodes of the graph
        cudaEvent_t e0 = pool[pool_used], e1 = pool[pool_used + 1];
        pool_used += 2;
        const unsigned int rf = use_graph ? cudaEventRecordExternal : cudaEventRecordDefault;
        cudaError_t e = cudaEventRecordWithFlags(e0, ctx->stream, rf);
        if (e == cudaSuccess)
            e = launch();
        if (e == cudaSuccess)
            e = cudaEventRecordWithFlags(e1, ctx->stream, rf);
        return e;
    };
    // programmatic dependent launch of the passes (never with per-pass events, whose record nodes sit
    // between the passes)
    const bool pdl = !timed && (ctx->pdl_mode == 1 || (ctx->pdl_mode < 0 && pdl_default(ctx)));
    DevPlace pp = ctx->place;
    pp.scen_warps = fused ? ctx->scen_warps : nullptr;
    auto pass = [&](int r, PassKind kind) -> cudaError_t {
        if (ctx->placement)
            return timed_launch([&]() { return launch_place(t, st, pp, a, r, kind, ctx->place_grid, ctx->stream); });
        // without per-pass events the previous operation is always a kernel: the pass overlaps its
        // start with that kernel's tail (programmatic dependent launch)
        return timed_launch([&]() { return launch_pass(t, st, pl, a, r, kind, ctx->grid, ctx->stream, pdl); });
    };
    auto issue = [&]() -> cudaError_t {
        cudaError_t e = launch_init(t, st, a, has_l0 ? ctx->lambda0 : nullptr, ctx->stream);
        if (place_res) {
            if (e == cudaSuccess && T > 0)
                e = timed_launch([&]() {
                    return hold ? launch_place_res_held(t, st, pp, a, ctx->place_res, ctx->stream)
                                : launch_place_res(t, st, pp, a, ctx->place_res, ctx->stream);
                });
            if (e == cudaSuccess)
                e = pass(T, PASS_FINAL);
            if (e == cudaSuccess)
                e = launch_objectives(t, st, a, ctx->stream);
            return e;
        }
        if (ri >= 0) {
            const ResPlan &rp = ctx->res[ri].plan;
            if (e == cudaSuccess)
                e = timed_launch([&]() { return launch_resident(t_orig, st, rp, a, ctx->stream); });
            if (e == cudaSuccess)
                e = launch_objectives(t, st, a, ctx->stream);
            return e;
        }
        if (persist) {
            if (e == cudaSuccess)
                e = launch_pass_persist(t, st, pl, a, T, ctx->persist_grid, ctx->stream);
            // after the cooperative launch the final pass starts as an ordinary launch
            if (e == cudaSuccess)
                e = launch_pass(t, st, pl, a, T, PASS_FINAL, ctx->grid, ctx->stream, false);
            if (e == cudaSuccess)
                e = launch_objectives(t, st, a, ctx->stream);
            return e;
        }
        for (int r = 0; r < T && e == cudaSuccess; ++r) {
            if (ctx->grid > 0)
                e = pass(r, PASS_ROUND);
            if (e == cudaSuccess && !fused)
                e = launch_update(t, st, a, r, ctx->stream);
        }
        if (e == cudaSuccess && ctx->grid > 0)
            e = pass(T, PASS_FINAL);
        if (e == cudaSuccess)
            e = launch_objectives(t, st, a, ctx->stream);
        return e;
    };
    ctx->last_launches = place_res ? 3 + (T > 0 ? 1 : 0)
                         : ri >= 0 ? 3
                         : persist ? 4
                                   : 3 + (fused ? 1LL : 2LL) * T - (ctx->grid > 0 ? 0 : (T + 1));
    ctx->last_T = T;

    GraphKey key;
    key.eta0 = p->eta0;
    key.tol = p->tol;
    key.step = p->step;
    key.mode = p->mode;
    key.T = T;
    key.flags = p->flags;
    key.lt = st.lam_trace;
    key.tt = st.time_trace;
    key.dt = st.dem_trace;
    key.ht = st.hash_trace;
    key.gt = st.dual_trace;
    key.has_l0 = has_l0;
    key.res = place_res ? -2 : ri;
    key.hold = hold;
    key.persist = persist;
    key.hold_tx = a.hold_tx;
    key.wait_ms = a.wait_ms;
    {
        // FNV-1a over the kernel arguments (structs built zero-padded) and launch shapes: a reload that
        // leaves every argument as it was (a table of the same shape: the buffer pool hands every
        // buffer back to its role) replays the previous graph as it is
        uint64_t h = 1469598103934665603ull;
        auto mix = [&](const void *p, size_t n) {
            const unsigned char *b = static_cast<const unsigned char *>(p);
            for (size_t i = 0; i < n; ++i)
                h = (h ^ b[i]) * 1099511628211ull;
        };
        mix(&t, sizeof(t));
        mix(&t_orig, sizeof(t_orig));
        mix(&st, sizeof(st));
        mix(&pl, sizeof(pl));
        mix(&a, sizeof(a));
        mix(&pp, sizeof(pp));
        mix(&ctx->lambda0, sizeof(ctx->lambda0));
        const int64_t shape[5] = {ctx->grid, ctx->persist_grid, ctx->place_grid, pdl ? 1 : 0, (int64_t)ri};
        mix(shape, sizeof(shape));
        if (ri >= 0)
            mix(&ctx->res[ri].plan, sizeof(ResPlan));
        if (place_res)
            mix(&ctx->place_res, sizeof(ctx->place_res));
        key.args = h;
    }

    if (!use_graph) {
        ESP_CUDA(record_solve_event(ctx, 0));
        ESP_CUDA(issue());
        ESP_CUDA(record_solve_event(ctx, 1));
        ctx->ev_used = pool_used;
        return ESP_OK;
    }
    if (!(ctx->gexec && ctx->gkey == key)) {
        cudaGraph_t g = nullptr;
        ESP_CUDA(cudaStreamBeginCapture(ctx->stream, cudaStreamCaptureModeThreadLocal));
        cudaError_t e = issue();
        cudaError_t e2 = cudaStreamEndCapture(ctx->stream, &g);
        if (e != cudaSuccess || e2 != cudaSuccess) {
            if (g)
                cudaGraphDestroy(g);
            return cuda_fail(ctx, e != cudaSuccess ? e : e2);
        }
        // the same launches with other arguments (a reload of the same shape, another eta0 or
        // tolerance): update the executable graph in place; else instantiate a new one
        bool updated = false;
        if (ctx->gexec) {
            cudaGraphExecUpdateResultInfo info;
            if (cudaGraphExecUpdate(ctx->gexec, g, &info) == cudaSuccess) {
                updated = true;
            } else {
                cudaGetLastError();
                cudaGraphExecDestroy(ctx->gexec);
                ctx->gexec = nullptr;
            }
        }
        if (!updated) {
            e = cudaGraphInstantiate(&ctx->gexec, g, 0);
            if (e != cudaSuccess) {
                cudaGraphDestroy(g);
                ctx->gexec = nullptr;
                return cuda_fail(ctx, e);
            }
        }
        cudaGraphDestroy(g);
        ctx->gkey = key;
        ctx->graph_pairs = timed ? pool_used / 2 : 0;
    }
    ESP_CUDA(record_solve_event(ctx, 0));
    ESP_CUDA(cudaGraphLaunch(ctx->gexec, ctx->stream));
    ESP_CUDA(record_solve_event(ctx, 1));
    if (timed)
        ctx->graph_timed_run = true;
    return ESP_OK;
}

esp_status read_results(esp_ctx *ctx, esp_result *out)
{
    const int S = ctx->S;
    std::vector<int32_t> rr(S), cv(S), ss(S), fe(S);
    std::vector<double> pr(S), du(S), bd(S);
    ESP_CUDA(cudaMemcpyAsync(rr.data(), ctx->rounds_run, S * 4, cudaMemcpyDeviceToHost, ctx->stream));
    ESP_CUDA(cudaMemcpyAsync(cv.data(), ctx->converged, S * 4, cudaMemcpyDeviceToHost, ctx->stream));
    ESP_CUDA(cudaMemcpyAsync(ss.data(), ctx->status, S * 4, cudaMemcpyDeviceToHost, ctx->stream));
    ESP_CUDA(cudaMemcpyAsync(fe.data(), ctx->feasible, S * 4, cudaMemcpyDeviceToHost, ctx->stream));
    ESP_CUDA(cudaMemcpyAsync(pr.data(), ctx->primal, S * 8, cudaMemcpyDeviceToHost, ctx->stream));
    ESP_CUDA(cudaMemcpyAsync(du.data(), ctx->dual, S * 8, cudaMemcpyDeviceToHost, ctx->stream));
    ESP_CUDA(cudaMemcpyAsync(bd.data(), ctx->best_dual, S * 8, cudaMemcpyDeviceToHost, ctx->stream));
    ESP_CUDA(cudaStreamSynchronize(ctx->stream));
    float ms = 0.0f;
    if (ctx->solve_timed && cudaEventElapsedTime(&ms, ctx->solve_ev[0], ctx->solve_ev[1]) != cudaSuccess) {
        cudaGetLastError();
        ms = 0.0f;
    }
    bool overflow = false;
    for (int s = 0; s < S; ++s) {
        out[s].device_ms = ms;
        out[s].rounds_run = rr[s];
        out[s].converged = cv[s];
        out[s].feasible = fe[s];
        out[s].status = ss[s] ? ESP_ERR_OVERFLOW : ESP_OK;
        out[s].primal = pr[s];
        out[s].dual = du[s];
        out[s].best_dual = bd[s];
        overflow |= ss[s] != 0;
    }
    return overflow ? ESP_ERR_OVERFLOW : ESP_OK;
}

esp_status check_device_error(esp_ctx *ctx)
{
    unsigned int e = 0;
    ESP_CUDA(cudaMemcpyAsync(&e, ctx->err, sizeof(e), cudaMemcpyDeviceToHost, ctx->stream));
    ESP_CUDA(cudaStreamSynchronize(ctx->stream));
    if (e & DEV_ERR_TIMEOUT) {
        ctx->poisoned = true;
        return ESP_ERR_TIMEOUT;
    }
    return ESP_OK;
}

}  // namespace

extern "C" {

const char *esp_status_string(esp_status s)
{
    switch (s) {
    case ESP_OK: return "ok";
    case ESP_ERR_INVALID_ARG: return "invalid argument";
    case ESP_ERR_OVERFLOW: return "overflow (a price became non-finite)";
    case ESP_ERR_OOM: return "out of memory";
    case ESP_ERR_CUDA: return "CUDA error";
    case ESP_ERR_NOT_LOADED: return "no table loaded / nothing solved";
    case ESP_ERR_TIMEOUT: return "device wait timed out";
    case ESP_ERR_STATE: return "context unusable after an earlier CUDA error or timeout";
    case ESP_ERR_UNSUPPORTED: return "unsupported device";
    }
    return "unknown status";
}

esp_status esp_create(esp_ctx **out, int device, void *cuda_stream)
{
    if (!out)
        return ESP_ERR_INVALID_ARG;
    *out = nullptr;
    int n = 0;
    if (cudaGetDeviceCount(&n) != cudaSuccess || n == 0) {
        cudaGetLastError();
        return ESP_ERR_UNSUPPORTED;
    }
    if (device < 0) {
        if (cudaGetDevice(&device) != cudaSuccess)
            return ESP_ERR_CUDA;
    }
    if (device >= n)
        return ESP_ERR_INVALID_ARG;
    cudaDeviceProp prop;
    if (cudaGetDeviceProperties(&prop, device) != cudaSuccess)
        return ESP_ERR_CUDA;
    if (prop.major != 10 || prop.minor != 3)
        return ESP_ERR_UNSUPPORTED;
    esp_ctx *ctx = new (std::nothrow) esp_ctx();
    if (!ctx)
        return ESP_ERR_OOM;
    ctx->device = device;
    ctx->stream = static_cast<cudaStream_t>(cuda_stream);
    ctx->sm_count = prop.multiProcessorCount;
    if (cudaSetDevice(device) != cudaSuccess) {
        delete ctx;
        return ESP_ERR_CUDA;
    }
    *out = ctx;
    return ESP_OK;
}

esp_status esp_set_stream(esp_ctx *ctx, void *cuda_stream)
{
    esp_status st = check_ctx(ctx);
    if (st != ESP_OK)
        return st;
    if (ctx->stream != static_cast<cudaStream_t>(cuda_stream)) {
        // work queued on the old stream finishes before another stream can reuse the buffers
        ESP_CUDA(cudaSetDevice(ctx->device));
        ESP_CUDA(cudaStreamSynchronize(ctx->stream));
        if (ctx->gexec) {
            cudaGraphExecDestroy(ctx->gexec);
            ctx->gexec = nullptr;
            ctx->gkey = GraphKey();
        }
    }
    ctx->stream = static_cast<cudaStream_t>(cuda_stream);
    return ESP_OK;
}

esp_status esp_load_options(esp_ctx *ctx, int32_t S, int32_t J, int32_t R, int32_t P, int32_t r_global,
                            const int64_t *job_offsets, const int32_t *units, const double *values,
                            const uint16_t *group, const int64_t *capacity)
{
    esp_status st = check_ctx(ctx);
    if (st != ESP_OK)
        return st;
    LoadStreamScope scope(ctx);
    if ((st = scope.begin()) != ESP_OK)
        return st;
    return load_common(ctx, S, J, R, P, r_global, job_offsets, units, values, group, capacity, false);
}

esp_status esp_load_options_device(esp_ctx *ctx, int32_t S, int32_t J, int32_t R, int32_t P, int32_t r_global,
                                   const int64_t *job_offsets, const int32_t *units, const double *values,
                                   const uint16_t *group, const int64_t *capacity)
{
    esp_status st = check_ctx(ctx);
    if (st != ESP_OK)
        return st;
    LoadStreamScope scope(ctx);
    if ((st = scope.begin()) != ESP_OK)
        return st;
    return load_common(ctx, S, J, R, P, r_global, job_offsets, units, values, group, capacity, true);
}

esp_status esp_solve_async(esp_ctx *ctx, const esp_params *params)
{
    esp_status st = check_ctx(ctx);
    if (st != ESP_OK)
        return st;
    if (!ctx->loaded)
        return ESP_ERR_NOT_LOADED;
    if ((st = check_params(ctx, params)) != ESP_OK)
        return st;
    if (params->lambda_trace || params->demand_trace || params->selhash_trace || params->dual_trace ||
        params->round_time_trace)
        return ESP_ERR_INVALID_ARG;
    ESP_CUDA(cudaSetDevice(ctx->device));
    const size_t SP = (size_t)ctx->S * ctx->P;
    if (params->lambda0)
        ESP_CUDA(cudaMemcpyAsync(ctx->lambda0, params->lambda0, SP * sizeof(double), cudaMemcpyHostToDevice,
                                 ctx->stream));
    const DevState ds = dev_state(ctx);
    if ((st = enqueue_solve(ctx, params, ds, params->lambda0 != nullptr)) != ESP_OK)
        return st;
    ctx->solved = true;
    return ESP_OK;
}

esp_status esp_solve(esp_ctx *ctx, const esp_params *params, esp_result *out)
{
    esp_status st = check_ctx(ctx);
    if (st != ESP_OK)
        return st;
    if (!ctx->loaded)
        return ESP_ERR_NOT_LOADED;
    if ((st = check_params(ctx, params)) != ESP_OK)
        return st;
    ESP_CUDA(cudaSetDevice(ctx->device));
    const size_t S = ctx->S, P = ctx->P, T = params->max_rounds;
    if (params->lambda0)
        ESP_CUDA(cudaMemcpyAsync(ctx->lambda0, params->lambda0, S * P * sizeof(double), cudaMemcpyHostToDevice,
                                 ctx->stream));
    DevState ds = dev_state(ctx);
    // traces: device copies start from the caller's contents, so rows never written stay as they were
    if (params->lambda_trace) {
        if ((st = grow(ctx, ctx->lt, S * (T + 1) * P)) != ESP_OK)
            return st;
        ESP_CUDA(cudaMemcpyAsync(ctx->lt.p, params->lambda_trace, S * (T + 1) * P * 8, cudaMemcpyHostToDevice,
                                 ctx->stream));
        ds.lam_trace = ctx->lt.p;
    }
    if (params->demand_trace && T > 0) {
        if ((st = grow(ctx, ctx->dt, S * T * P)) != ESP_OK)
            return st;
        ESP_CUDA(cudaMemcpyAsync(ctx->dt.p, params->demand_trace, S * T * P * 8, cudaMemcpyHostToDevice,
                                 ctx->stream));
        ds.dem_trace = ctx->dt.p;
    }
    if (params->selhash_trace && T > 0) {
        if ((st = grow(ctx, ctx->ht, S * T)) != ESP_OK)
            return st;
        ESP_CUDA(cudaMemcpyAsync(ctx->ht.p, params->selhash_trace, S * T * 8, cudaMemcpyHostToDevice, ctx->stream));
        ds.hash_trace = ctx->ht.p;
    }
    if (params->dual_trace) {
        if ((st = grow(ctx, ctx->gt, S * (T + 1))) != ESP_OK)
            return st;
        ESP_CUDA(cudaMemcpyAsync(ctx->gt.p, params->dual_trace, S * (T + 1) * 8, cudaMemcpyHostToDevice, ctx->stream));
        ds.dual_trace = ctx->gt.p;
    }
    if (params->round_time_trace && T > 0) {
        if ((st = grow(ctx, ctx->tt, S * T)) != ESP_OK)
            return st;
        ESP_CUDA(cudaMemcpyAsync(ctx->tt.p, params->round_time_trace, S * T * 8, cudaMemcpyHostToDevice,
                                 ctx->stream));
        ds.time_trace = ctx->tt.p;
    }
    if ((st = enqueue_solve(ctx, params, ds, params->lambda0 != nullptr)) != ESP_OK)
        return st;
    ctx->solved = true;
    if ((st = check_device_error(ctx)) != ESP_OK)
        return st;
    if (params->lambda_trace)
        ESP_CUDA(cudaMemcpyAsync(params->lambda_trace, ctx->lt.p, S * (T + 1) * P * 8, cudaMemcpyDeviceToHost,
                                 ctx->stream));
    if (ds.dem_trace)
        ESP_CUDA(cudaMemcpyAsync(params->demand_trace, ctx->dt.p, S * T * P * 8, cudaMemcpyDeviceToHost, ctx->stream));
    if (ds.hash_trace)
        ESP_CUDA(cudaMemcpyAsync(params->selhash_trace, ctx->ht.p, S * T * 8, cudaMemcpyDeviceToHost, ctx->stream));
    if (params->dual_trace)
        ESP_CUDA(cudaMemcpyAsync(params->dual_trace, ctx->gt.p, S * (T + 1) * 8, cudaMemcpyDeviceToHost, ctx->stream));
    if (ds.time_trace)
        ESP_CUDA(cudaMemcpyAsync(params->round_time_trace, ctx->tt.p, S * T * 8, cudaMemcpyDeviceToHost,
                                 ctx->stream));
    if (out)
        return read_results(ctx, out);
    ESP_CUDA(cudaStreamSynchronize(ctx->stream));
    return ESP_OK;
}

esp_status esp_get_result(esp_ctx *ctx, esp_result *out)
{
    esp_status st = check_ctx(ctx);
    if (st != ESP_OK)
        return st;
    if (!out)
        return ESP_ERR_INVALID_ARG;
    if (!ctx->solved)
        return ESP_ERR_NOT_LOADED;
    if ((st = check_device_error(ctx)) != ESP_OK)
        return st;
    return read_results(ctx, out);
}

static esp_status get_array(esp_ctx *ctx, void *out, const void *src, size_t bytes)
{
    esp_status st = check_ctx(ctx);
    if (st != ESP_OK)
        return st;
    if (!out)
        return ESP_ERR_INVALID_ARG;
    if (!ctx->solved)
        return ESP_ERR_NOT_LOADED;
    if ((st = check_device_error(ctx)) != ESP_OK)
        return st;
    ESP_CUDA(cudaMemcpyAsync(out, src, bytes, cudaMemcpyDeviceToHost, ctx->stream));
    ESP_CUDA(cudaStreamSynchronize(ctx->stream));
    return ESP_OK;
}

esp_status esp_get_prices(esp_ctx *ctx, double *out)
{
    if (!ctx)
        return ESP_ERR_INVALID_ARG;
    return get_array(ctx, out, ctx->lam, (size_t)ctx->S * ctx->P * sizeof(double));
}

esp_status esp_get_selection(esp_ctx *ctx, int32_t *out)
{
    if (!ctx)
        return ESP_ERR_INVALID_ARG;
    return get_array(ctx, out, ctx->sel, (size_t)ctx->S * ctx->J * sizeof(int32_t));
}

esp_status esp_get_demand(esp_ctx *ctx, int64_t *out)
{
    if (!ctx)
        return ESP_ERR_INVALID_ARG;
    return get_array(ctx, out, ctx->U_final, (size_t)ctx->S * ctx->P * sizeof(int64_t));
}

esp_status esp_evaluate(esp_ctx *ctx, const double *lambda, int32_t mode, uint32_t flags, int32_t *sel,
                        int64_t *demand, double *min_score)
{
    esp_status st = check_ctx(ctx);
    if (st != ESP_OK)
        return st;
    if (!ctx->loaded)
        return ESP_ERR_NOT_LOADED;
    if (!lambda || (mode != ESP_PRICE_RAW && mode != ESP_PRICE_NORMALIZED) || (flags & ~ESP_FLAG_EXACT_ONLY))
        return ESP_ERR_INVALID_ARG;
    const size_t SP = (size_t)ctx->S * ctx->P, SJ = (size_t)ctx->S * ctx->J;
    for (size_t i = 0; i < SP; ++i)
        if (!(lambda[i] >= 0.0) || !std::isfinite(lambda[i]))
            return ESP_ERR_INVALID_ARG;
    ESP_CUDA(cudaSetDevice(ctx->device));
    if (!state_ready(ctx))
        return ESP_ERR_STATE;
    ESP_CUDA(cudaMemcpyAsync(ctx->lambda0, lambda, SP * sizeof(double), cudaMemcpyHostToDevice, ctx->stream));
    const DevTable t = pass_table(ctx);
    DevState ds = dev_state(ctx);
    const DevPlan pl = dev_plan(ctx, false);
    const SolveArgs a = solve_args(ctx, 1.0, 0, mode, 0, 0.0, flags);
    ESP_CUDA(record_solve_event(ctx, 0));
    ESP_CUDA(launch_init(t, ds, a, ctx->lambda0, ctx->stream));
    if (ctx->placement)
        ESP_CUDA(launch_place(t, ds, ctx->place, a, 0, PASS_FINAL, ctx->place_grid, ctx->stream));
    else if (ctx->grid > 0)
        ESP_CUDA(launch_pass(t, ds, pl, a, 0, PASS_FINAL, ctx->grid, ctx->stream));
    ESP_CUDA(launch_objectives(t, ds, a, ctx->stream));
    ESP_CUDA(record_solve_event(ctx, 1));
    ctx->solved = true;
    if ((st = check_device_error(ctx)) != ESP_OK)
        return st;
    if (sel)
        ESP_CUDA(cudaMemcpyAsync(sel, ctx->sel, SJ * 4, cudaMemcpyDeviceToHost, ctx->stream));
    if (demand)
        ESP_CUDA(cudaMemcpyAsync(demand, ctx->U_final, SP * 8, cudaMemcpyDeviceToHost, ctx->stream));
    if (min_score)
        ESP_CUDA(cudaMemcpyAsync(min_score, ctx->job_min, SJ * 8, cudaMemcpyDeviceToHost, ctx->stream));
    ESP_CUDA(cudaStreamSynchronize(ctx->stream));
    return ESP_OK;
}

esp_status esp_load_placement(esp_ctx *ctx, int32_t S, int32_t J, int32_t KC, int32_t N, int32_t R, int32_t r_global,
                              const int32_t *cfg_units, const double *cfg_values, const float *sens,
                              const int32_t *job_type, int32_t NT, const int32_t *node_type, const float *D,
                              const int64_t *capacity)
{
    esp_status st = check_ctx(ctx);
    if (st != ESP_OK)
        return st;
    if (S < 1 || J < 1 || KC < 1 || KC > kPlaceMaxKC || N < 1 || N > kPlaceMaxN || R < 1 || R > kMaxR ||
        r_global < 0 || r_global >= R || NT < 1 || NT > kPlaceMaxNT || !cfg_units || !cfg_values || !sens ||
        !job_type || !node_type || !D || !capacity)
        return ESP_ERR_INVALID_ARG;
    const int64_t n_jobs = (int64_t)S * J;
    const int32_t P = r_global + (R - r_global) * N;
    if (n_jobs >= INT32_MAX)
        return ESP_ERR_INVALID_ARG;
    // validation and the per-scenario maxima on the host (the factored table is small)
    double dmax = 0.0;
    for (int32_t i = 0; i < NT * NT; ++i) {
        if (!std::isfinite(D[i]))
            return ESP_ERR_INVALID_ARG;
        dmax = std::max(dmax, (double)std::fabs(D[i]));
    }
    for (int32_t n = 0; n < N; ++n)
        if (node_type[n] < 0 || node_type[n] >= NT)
            return ESP_ERR_INVALID_ARG;
    for (int64_t i = 0; i < (int64_t)S * P; ++i)
        if (capacity[i] <= 0)
            return ESP_ERR_INVALID_ARG;
    std::vector<double> vmax((size_t)S, 0.0);
    std::vector<int32_t> umax((size_t)S * R, 0);
    std::vector<uint32_t> dup((size_t)n_jobs, 0u);
    int32_t small = 1;
    for (int64_t j = 0; j < n_jobs; ++j) {
        const int64_t s = j / J;
        if (!std::isfinite(sens[j]) || job_type[j] < 0 || job_type[j] >= NT)
            return ESP_ERR_INVALID_ARG;
        double vm = 0.0;
        for (int32_t k = 0; k < KC; ++k) {
            const double v = cfg_values[j * KC + k];
            if (!std::isfinite(v))
                return ESP_ERR_INVALID_ARG;
            vm = std::max(vm, std::fabs(v));
            const int32_t *u = cfg_units + (j * KC + k) * R;
            for (int32_t r = 0; r < R; ++r) {
                if (u[r] < 0)
                    return ESP_ERR_INVALID_ARG;
                umax[(size_t)s * R + r] = std::max(umax[(size_t)s * R + r], u[r]);
                if (u[r] >= (1 << 23))
                    small = 0;
            }
            for (int32_t k2 = 0; k2 < k; ++k2) {   // configuration k repeats configuration k2
                if (std::memcmp(&cfg_values[j * KC + k2], &v, sizeof(double)) == 0 &&
                    std::memcmp(cfg_units + (j * KC + k2) * R, u, sizeof(int32_t) * (size_t)R) == 0) {
                    dup[(size_t)j] |= 1u << k;
                    break;
                }
            }
        }
        // |v_kn| <= |v_k| + |sens * D| (the fp32 product rounds by at most 2^-24 relative)
        const double bound = vm + std::fabs((double)sens[j]) * dmax * (1.0 + 0x1p-20);
        vmax[(size_t)s] = std::max(vmax[(size_t)s], bound);
    }
    const int smem = place_smem_bytes(R, P, KC, N, NT);
    int optin = 0;
    ESP_CUDA(cudaSetDevice(ctx->device));
    ESP_CUDA(cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, ctx->device));
    if (smem > optin)
        return ESP_ERR_UNSUPPORTED;
    const int per_sm = place_ctas_per_sm(R, P, KC, N, NT);
    if (per_sm < 1)
        return ESP_ERR_UNSUPPORTED;
    release_table(ctx, true);
    ctx->S = S;
    ctx->J = J;
    ctx->R = R;
    ctx->P = P;
    ctx->rg = r_global;
    ctx->n_groups = N;
    ctx->n_opt = n_jobs * KC * N;
    ctx->small_units = small;
    ctx->placement = true;

    // warps: contiguous job ranges; the warps touching a scenario arrive once for its price update
    const int32_t W = (int32_t)std::min<int64_t>(n_jobs, (int64_t)ctx->sm_count * per_sm * kPlaceWarps);
    std::vector<int32_t> wj((size_t)W + 1), sw((size_t)S, 0);
    for (int32_t w = 0; w <= W; ++w)
        wj[(size_t)w] = (int32_t)((__int128)n_jobs * w / W);
    for (int32_t w = 0; w < W; ++w)
        if (wj[w + 1] > wj[w])
            for (int64_t sc = wj[w] / J; sc <= (wj[w + 1] - 1) / J; ++sc)
                ++sw[(size_t)sc];

#define PALLOC(ptr, count)                                \
    do {                                                  \
        esp_status a_ = dev_alloc(ctx, &(ptr), (count));  \
        if (a_ != ESP_OK) {                               \
            release_table(ctx);                           \
            return a_;                                    \
        }                                                 \
    } while (0)
    int32_t *d_units = nullptr, *d_jt = nullptr, *d_nt = nullptr, *d_wj = nullptr;
    double *d_vals = nullptr;
    float *d_sens = nullptr, *d_D = nullptr;
    uint32_t *d_dup = nullptr;
    PALLOC(d_units, (size_t)n_jobs * KC * R);
    PALLOC(d_vals, (size_t)n_jobs * KC);
    PALLOC(d_sens, (size_t)n_jobs);
    PALLOC(d_jt, (size_t)n_jobs);
    PALLOC(d_nt, (size_t)N);
    PALLOC(d_D, (size_t)NT * NT);
    PALLOC(d_dup, (size_t)n_jobs);
    PALLOC(d_wj, (size_t)W + 1);
    PALLOC(ctx->scen_warps, (size_t)S);
    PALLOC(ctx->arrive, (size_t)S);
    PALLOC(ctx->cap, (size_t)S * P);
    PALLOC(ctx->vmax, (size_t)S);
    PALLOC(ctx->umax, (size_t)S * R);
    PALLOC(ctx->valflags, 4);
    PALLOC(ctx->stats, 4);
    auto h2d = [&](void *dst, const void *src, size_t bytes) {
        return cudaMemcpyAsync(dst, src, bytes, cudaMemcpyHostToDevice, ctx->stream);
    };
    ESP_CUDA(h2d(d_units, cfg_units, (size_t)n_jobs * KC * R * sizeof(int32_t)));
    ESP_CUDA(h2d(d_vals, cfg_values, (size_t)n_jobs * KC * sizeof(double)));
    ESP_CUDA(h2d(d_sens, sens, (size_t)n_jobs * sizeof(float)));
    ESP_CUDA(h2d(d_jt, job_type, (size_t)n_jobs * sizeof(int32_t)));
    ESP_CUDA(h2d(d_nt, node_type, (size_t)N * sizeof(int32_t)));
    ESP_CUDA(h2d(d_D, D, (size_t)NT * NT * sizeof(float)));
    ESP_CUDA(h2d(d_dup, dup.data(), dup.size() * sizeof(uint32_t)));
    ESP_CUDA(h2d(d_wj, wj.data(), wj.size() * sizeof(int32_t)));
    ESP_CUDA(h2d(ctx->scen_warps, sw.data(), sw.size() * sizeof(int32_t)));
    ESP_CUDA(h2d(ctx->cap, capacity, (size_t)S * P * sizeof(int64_t)));
    ESP_CUDA(h2d(ctx->vmax, vmax.data(), vmax.size() * sizeof(double)));
    ESP_CUDA(h2d(ctx->umax, umax.data(), umax.size() * sizeof(int32_t)));
    ctx->place.cfg_units = d_units;
    ctx->place.cfg_values = d_vals;
    ctx->place.sens = d_sens;
    ctx->place.job_type = d_jt;
    ctx->place.node_type = d_nt;
    ctx->place.D = d_D;
    ctx->place.cfg_dup = d_dup;
    ctx->place.warp_job = d_wj;
    ctx->place.scen_warps = nullptr;
    ctx->place.KC = KC;
    ctx->place.N = N;
    ctx->place.NT = NT;
    ctx->place.n_warps = W;
    ctx->place_grid = (W + kPlaceWarps - 1) / kPlaceWarps;
    ctx->grid = ctx->place_grid;
    if ((st = alloc_solve_state(ctx)) != ESP_OK) {
        release_table(ctx);
        return st;
    }
    // the grid-resident solve (ESP_FLAG_RESIDENT): one CTA per SM holds the price state of every
    // scenario and each warp at most kPlaceResJobs jobs, all in shared memory
    if ((int64_t)S * P <= kPlaceResMaxPrices &&
        n_jobs <= (int64_t)kPlaceResJobs * kPlaceResWarps * ctx->sm_count &&
        place_res_smem_bytes(S, P, KC, R) <= optin && place_res_ctas_per_sm(S, P, KC, R) >= 1) {
        PlaceRes &pr = ctx->place_res;
        const int32_t Wr = (int32_t)std::min<int64_t>(n_jobs, (int64_t)kPlaceResWarps * ctx->sm_count);
        std::vector<int32_t> wr((size_t)Wr + 1);
        for (int32_t w = 0; w <= Wr; ++w)
            wr[(size_t)w] = (int32_t)((__int128)n_jobs * w / Wr);
        int32_t *d_wr = nullptr;
        PALLOC(pr.U3, 3 * (size_t)S * P);
        PALLOC(pr.bar, 2);
        PALLOC(d_wr, (size_t)Wr + 1);
        ESP_CUDA(h2d(d_wr, wr.data(), wr.size() * sizeof(int32_t)));
        pr.warp_job = d_wr;
        pr.n_warps = Wr;
        pr.grid = (Wr + kPlaceResWarps - 1) / kPlaceResWarps;
        ctx->place_res_ok = true;
    }
#undef PALLOC
    ESP_CUDA(cudaStreamSynchronize(ctx->stream));
    trim_pool(ctx);
    ctx->loaded = true;
    ctx->solved = false;
    return ESP_OK;
}

namespace {

// After the values changed: clear and redo the duplicate marks, the per-scenario maxima (and the
// validation they come with) and the sorted copy. Returns the validation flags.
esp_status refresh_after_values(esp_ctx *ctx, unsigned int *vflags)
{
    const DevTable t = dev_table(ctx);
    ESP_CUDA(launch_clear_marks(ctx->units, ctx->n_opt, ctx->R, ctx->stream));
    ESP_CUDA(cudaMemsetAsync(ctx->vmax, 0, (size_t)ctx->S * sizeof(double), ctx->stream));
    ESP_CUDA(cudaMemsetAsync(ctx->umax, 0, (size_t)ctx->S * ctx->R * sizeof(int32_t), ctx->stream));
    ESP_CUDA(cudaMemsetAsync(ctx->valflags, 0, sizeof(unsigned int), ctx->stream));
    ESP_CUDA(launch_validate(t, ctx->vmax, ctx->umax, ctx->valflags, ctx->stream));
    ESP_CUDA(cudaMemsetAsync(ctx->stats + 1, 0, sizeof(unsigned long long), ctx->stream));
    ESP_CUDA(launch_mark_duplicates(t, ctx->units, ctx->stats + 1, ctx->stream, ctx->max_k));
    if (ctx->sorted)
        ESP_CUDA(launch_gather_sorted(t, pass_table(ctx), ctx->s_units, ctx->s_values, ctx->stream));
    if (ctx->il)
        ESP_CUDA(launch_interleave(pass_table(ctx), ctx->tiles, ctx->n_tiles, ctx->il, ctx->il_f32, ctx->stream));
    ESP_CUDA(cudaMemcpyAsync(vflags, ctx->valflags, sizeof(unsigned int), cudaMemcpyDeviceToHost, ctx->stream));
    ESP_CUDA(cudaStreamSynchronize(ctx->stream));
    return ESP_OK;
}

}  // namespace

esp_status esp_set_penalties(esp_ctx *ctx, double gamma0, const int32_t *c_cur, double alpha, const double *s_hat,
                             const double *tau)
{
    esp_status st = check_ctx(ctx);
    if (st != ESP_OK)
        return st;
    if (!ctx->loaded)
        return ESP_ERR_NOT_LOADED;
    if (ctx->placement)
        return ESP_ERR_UNSUPPORTED;
    if (!(gamma0 >= 0.0) || !std::isfinite(gamma0) || !(alpha >= 0.0) || !std::isfinite(alpha) || (s_hat && !tau))
        return ESP_ERR_INVALID_ARG;
    ESP_CUDA(cudaSetDevice(ctx->device));
    const size_t n_jobs = (size_t)ctx->S * ctx->J, n_opt = (size_t)ctx->n_opt;
    if (!ctx->values0) {
        void *q = nullptr;
        cudaError_t e = cudaMalloc(&q, n_opt * sizeof(double) + 64);
        if (e == cudaErrorMemoryAllocation) {
            cudaGetLastError();
            return ESP_ERR_OOM;
        }
        ESP_CUDA(e);
        ctx->table_bufs.emplace_back(q, n_opt * sizeof(double) + 64);
        ctx->values0 = static_cast<double *>(q);
        ESP_CUDA(cudaMemcpyAsync(ctx->values0, ctx->values, n_opt * sizeof(double), cudaMemcpyDeviceToDevice,
                                 ctx->stream));
    }
    // inputs on the device, for this call only
    void *buf = nullptr;
    const size_t cur_b = c_cur ? n_jobs * sizeof(int32_t) : 0, sh_b = s_hat ? n_opt * sizeof(double) : 0,
                 tau_b = s_hat ? n_jobs * sizeof(double) : 0;
    const size_t a1 = (cur_b + 255) & ~size_t(255), a2 = (sh_b + 255) & ~size_t(255);
    if (cur_b + sh_b + tau_b > 0) {
        cudaError_t e = cudaMalloc(&buf, a1 + a2 + tau_b + 64);
        if (e == cudaErrorMemoryAllocation) {
            cudaGetLastError();
            return ESP_ERR_OOM;
        }
        ESP_CUDA(e);
    }
    unsigned char *b = static_cast<unsigned char *>(buf);
    int32_t *d_cur = c_cur ? reinterpret_cast<int32_t *>(b) : nullptr;
    double *d_sh = s_hat ? reinterpret_cast<double *>(b + a1) : nullptr;
    double *d_tau = s_hat ? reinterpret_cast<double *>(b + a1 + a2) : nullptr;
    auto done = [&](esp_status r) {
        if (buf) {
            cudaStreamSynchronize(ctx->stream);
            cudaFree(buf);
        }
        return r;
    };
#define ESP_PEN_CUDA(call)                          \
    do {                                            \
        cudaError_t e_ = (call);                    \
        if (e_ != cudaSuccess) {                    \
            cudaGetLastError();                     \
            return done(cuda_fail(ctx, e_));        \
        }                                           \
    } while (0)
    if (c_cur)
        ESP_PEN_CUDA(cudaMemcpyAsync(d_cur, c_cur, cur_b, cudaMemcpyHostToDevice, ctx->stream));
    if (s_hat) {
        ESP_PEN_CUDA(cudaMemcpyAsync(d_sh, s_hat, sh_b, cudaMemcpyHostToDevice, ctx->stream));
        ESP_PEN_CUDA(cudaMemcpyAsync(d_tau, tau, tau_b, cudaMemcpyHostToDevice, ctx->stream));
    }
    ESP_PEN_CUDA(cudaMemsetAsync(ctx->valflags, 0, sizeof(unsigned int), ctx->stream));
    ESP_PEN_CUDA(launch_apply_penalties(dev_table(ctx), ctx->values0, d_cur, d_sh, d_tau, gamma0, alpha, ctx->values,
                                        ctx->valflags, ctx->stream));
    unsigned int pflags = 0;
    ESP_PEN_CUDA(cudaMemcpyAsync(&pflags, ctx->valflags, sizeof(unsigned int), cudaMemcpyDeviceToHost, ctx->stream));
    ESP_PEN_CUDA(cudaStreamSynchronize(ctx->stream));
#undef ESP_PEN_CUDA
    if (pflags) {   // back to the loaded values
        cudaError_t e = cudaMemcpyAsync(ctx->values, ctx->values0, n_opt * sizeof(double), cudaMemcpyDeviceToDevice,
                                        ctx->stream);
        if (e != cudaSuccess)
            return done(cuda_fail(ctx, e));
    }
    unsigned int vflags = 0;
    st = refresh_after_values(ctx, &vflags);
    if (st != ESP_OK)
        return done(st);
    ctx->solved = false;
    return done((pflags || vflags) ? ESP_ERR_INVALID_ARG : ESP_OK);
}

esp_status esp_last_launch_count(esp_ctx *ctx, int64_t *out)
{
    if (!ctx || !out)
        return ESP_ERR_INVALID_ARG;
    *out = ctx->last_launches;
    return ESP_OK;
}

esp_status esp_pass_times(esp_ctx *ctx, double *total_ms, int64_t *count, int32_t reset)
{
    esp_status st = check_ctx(ctx);
    if (st != ESP_OK)
        return st;
    if (!total_ms || !count)
        return ESP_ERR_INVALID_ARG;
    ESP_CUDA(cudaStreamSynchronize(ctx->stream));
    double sum = 0.0;
    int64_t n = 0;
    for (size_t i = 0; i + 1 < ctx->ev_used; i += 2, ++n) {
        float ms = 0.0f;
        ESP_CUDA(cudaEventElapsedTime(&ms, ctx->ev_pool[i], ctx->ev_pool[i + 1]));
        sum += ms;
    }
    if (ctx->graph_timed_run) {   // the latest replay of the timed graph
        for (size_t i = 0; i < ctx->graph_pairs; ++i, ++n) {
            float ms = 0.0f;
            ESP_CUDA(cudaEventElapsedTime(&ms, ctx->graph_pool[2 * i], ctx->graph_pool[2 * i + 1]));
            sum += ms;
        }
    }
    *total_ms = sum;
    *count = n;
    if (reset) {
        ctx->ev_used = 0;
        ctx->graph_timed_run = false;
    }
    return ESP_OK;
}

void esp_destroy(esp_ctx *ctx)
{
    if (!ctx)
        return;
    cudaSetDevice(ctx->device);
    if (!ctx->poisoned)
        cudaStreamSynchronize(ctx->stream);
    release_table(ctx);
    if (ctx->lt.p) cudaFree(ctx->lt.p);
    if (ctx->dt.p) cudaFree(ctx->dt.p);
    if (ctx->ht.p) cudaFree(ctx->ht.p);
    if (ctx->gt.p) cudaFree(ctx->gt.p);
    if (ctx->tt.p) cudaFree(ctx->tt.p);
    for (cudaEvent_t e : ctx->ev_pool)
        cudaEventDestroy(e);
    for (cudaEvent_t e : ctx->graph_pool)
        cudaEventDestroy(e);
    for (cudaEvent_t e : ctx->solve_ev)
        if (e)
            cudaEventDestroy(e);
    if (ctx->load_stream) {
        cudaStreamSynchronize(ctx->load_stream);
        cudaStreamDestroy(ctx->load_stream);
    }
    if (ctx->h_stage)
        cudaFreeHost(ctx->h_stage);
    for (cudaEvent_t e : ctx->load_ev)
        if (e)
            cudaEventDestroy(e);
    delete ctx;
}

esp_status esp_debug_stats(esp_ctx *ctx, int64_t *resolutions, int64_t *marked, int32_t reset)
{
    esp_status st = check_ctx(ctx);
    if (st != ESP_OK)
        return st;
    if (!ctx->loaded || !resolutions || !marked)
        return ESP_ERR_INVALID_ARG;
    unsigned long long h[2] = {0, 0};
    ESP_CUDA(cudaMemcpyAsync(h, ctx->stats, sizeof(h), cudaMemcpyDeviceToHost, ctx->stream));
    ESP_CUDA(cudaStreamSynchronize(ctx->stream));
    *resolutions = (int64_t)h[0];
    *marked = (int64_t)h[1];
    if (reset)
        ESP_CUDA(cudaMemsetAsync(ctx->stats, 0, sizeof(unsigned long long), ctx->stream));
    return ESP_OK;
}

esp_status esp_debug_load_profile(esp_ctx *ctx, double *ms, int64_t *mallocs, int64_t *frees)
{
    esp_status st = check_ctx(ctx);
    if (st != ESP_OK)
        return st;
    if (!ms || !mallocs || !frees)
        return ESP_ERR_INVALID_ARG;
    for (int i = 0; i < 7; ++i)
        ms[i] = ctx->load_ms[i];
    *mallocs = ctx->load_mallocs;
    *frees = ctx->load_frees;
    return ESP_OK;
}

esp_status esp_debug_persist_waits(esp_ctx *ctx, int64_t *ns, int64_t *waits, int32_t reset)
{
    esp_status st = check_ctx(ctx);
    if (st != ESP_OK)
        return st;
    if (!ctx->loaded || !ns || !waits)
        return ESP_ERR_INVALID_ARG;
    unsigned long long h[2] = {0, 0};
    ESP_CUDA(cudaMemcpyAsync(h, ctx->stats + 2, sizeof(h), cudaMemcpyDeviceToHost, ctx->stream));
    ESP_CUDA(cudaStreamSynchronize(ctx->stream));
    *ns = (int64_t)h[0];
    *waits = (int64_t)h[1];
    if (reset)
        ESP_CUDA(cudaMemsetAsync(ctx->stats + 2, 0, sizeof(h), ctx->stream));
    return ESP_OK;
}

int32_t esp_debug_tile_options(int32_t R, int32_t grouped)
{
    return tile_options(R, grouped != 0);
}

esp_status esp_debug_resident(esp_ctx *ctx, int32_t force_cs, int32_t *cs, int32_t *clusters)
{
    esp_status st = check_ctx(ctx);
    if (st != ESP_OK)
        return st;
    if (!ctx->loaded)
        return ESP_ERR_NOT_LOADED;
    if (!ctx->placement && (st = plan_resident_options(ctx)) != ESP_OK)
        return st;
    if (ctx->res.empty())
        return ESP_ERR_UNSUPPORTED;
    if (force_cs != 0) {
        int found = -1;
        for (size_t i = 0; i < ctx->res.size(); ++i)
            if (ctx->res[i].plan.cs == force_cs)
                found = (int)i;
        if (found < 0)
            return ESP_ERR_INVALID_ARG;
        ctx->res_force = found;
    } else {
        ctx->res_force = -1;
    }
    const esp_ctx::ResOption &o = ctx->res[ctx->res_force >= 0 ? ctx->res_force : ctx->res_auto];
    if (cs)
        *cs = o.plan.cs;
    if (clusters)
        *clusters = o.clusters;
    return ESP_OK;
}

namespace {

esp_status export_plan(const Plan &p, int32_t *tiles, int32_t tiles_cap, int32_t *warp_begin, int32_t warps_cap,
                       int32_t *n_tiles, int32_t *n_warps)
{
    *n_tiles = (int32_t)p.tiles.size();
    *n_warps = p.n_warps;
    if ((int32_t)p.tiles.size() > tiles_cap || p.n_warps + 1 > warps_cap + 1 || !tiles || !warp_begin)
        return ESP_ERR_OOM;
    for (size_t i = 0; i < p.tiles.size(); ++i) {
        const TileDesc &d = p.tiles[i];
        int32_t *w = tiles + 8 * i;
        w[0] = (int32_t)(uint32_t)(d.opt_begin & 0xffffffff);
        w[1] = (int32_t)(d.opt_begin >> 32);
        w[2] = (int32_t)(uint32_t)(d.job_begin & 0xffffffff);
        w[3] = (int32_t)(d.job_begin >> 32);
        w[4] = d.n_opt;
        w[5] = d.n_job;
        w[6] = d.scenario;
        w[7] = (int32_t)d.flags;
    }
    for (int32_t w = 0; w <= p.n_warps; ++w)
        warp_begin[w] = p.warp_begin[w];
    return ESP_OK;
}

}  // namespace

esp_status esp_debug_plan(const int64_t *job_offsets, int32_t S, int32_t J, int32_t tile_opt, int32_t max_warps,
                          int32_t *tiles, int32_t tiles_cap, int32_t *warp_begin, int32_t warps_cap,
                          int32_t *n_tiles, int32_t *n_warps)
{
    if (!job_offsets || S < 1 || J < 0 || !n_tiles || !n_warps)
        return ESP_ERR_INVALID_ARG;
    Plan p;
    if (!plan_tiles(job_offsets, S, J, tile_opt, max_warps, p) || !check_plan(job_offsets, S, J, p))
        return ESP_ERR_INVALID_ARG;
    return export_plan(p, tiles, tiles_cap, warp_begin, warps_cap, n_tiles, n_warps);
}

esp_status esp_debug_plan_runs(const int64_t *off, const int32_t *scen, const int32_t *runk, int32_t S, int32_t J,
                               int32_t tile_opt, int32_t max_warps, int32_t *tiles, int32_t tiles_cap,
                               int32_t *warp_begin, int32_t warps_cap, int32_t *n_tiles, int32_t *n_warps)
{
    if (!off || !scen || !runk || S < 1 || J < 0 || !n_tiles || !n_warps)
        return ESP_ERR_INVALID_ARG;
    Plan p;
    if (!plan_tiles(off, S, J, tile_opt, max_warps, p, scen, runk) || !check_plan(off, S, J, p, scen, runk))
        return ESP_ERR_INVALID_ARG;
    return export_plan(p, tiles, tiles_cap, warp_begin, warps_cap, n_tiles, n_warps);
}

esp_status esp_debug_sort_layout(const int64_t *job_offsets, int32_t S, int32_t J, int64_t *off, int32_t *jmap,
                                 int32_t *scen, int32_t *runk)
{
    if (!job_offsets || !off || !jmap || !scen || !runk || S < 1 || J < 1)
        return ESP_ERR_INVALID_ARG;
    SortedLayout lay;
    if (!sort_layout(job_offsets, S, J, lay))
        return ESP_ERR_INVALID_ARG;
    std::memcpy(off, lay.off.data(), lay.off.size() * sizeof(int64_t));
    std::memcpy(jmap, lay.jmap.data(), lay.jmap.size() * sizeof(int32_t));
    std::memcpy(scen, lay.scen.data(), lay.scen.size() * sizeof(int32_t));
    std::memcpy(runk, lay.runk.data(), lay.runk.size() * sizeof(int32_t));
    return ESP_OK;
}

esp_status esp_debug_set_sorted_layout(esp_ctx *ctx, int32_t enable)
{
    esp_status st = check_ctx(ctx);
    if (st != ESP_OK)
        return st;
    ctx->sorted_enabled = enable != 0;
    return ESP_OK;
}

esp_status esp_debug_set_plan_waves(esp_ctx *ctx, int32_t waves)
{
    esp_status st = check_ctx(ctx);
    if (st != ESP_OK)
        return st;
    if (waves < 0 || waves > 8)
        return ESP_ERR_INVALID_ARG;
    ctx->plan_waves = waves;
    return ESP_OK;
}

esp_status esp_debug_set_pdl(esp_ctx *ctx, int32_t mode)
{
    esp_status st = check_ctx(ctx);
    if (st != ESP_OK)
        return st;
    if (mode < -1 || mode > 1)
        return ESP_ERR_INVALID_ARG;
    ctx->pdl_mode = mode;
    if (ctx->gexec) {   // the graph holds the launches of the previous setting
        cudaGraphExecDestroy(ctx->gexec);
        ctx->gexec = nullptr;
        ctx->gkey = GraphKey();
    }
    return ESP_OK;
}

esp_status esp_debug_set_wait_limit(esp_ctx *ctx, uint32_t limit_ms)
{
    esp_status st = check_ctx(ctx);
    if (st != ESP_OK)
        return st;
    ctx->wait_ms = limit_ms;
    return ESP_OK;
}

esp_status esp_debug_hold_stage(esp_ctx *ctx)
{
    esp_status st = check_ctx(ctx);
    if (st != ESP_OK)
        return st;
    if (!ctx->loaded || ctx->placement || ctx->grid == 0)
        return ESP_ERR_UNSUPPORTED;
    ctx->hold_tx = 16;
    return ESP_OK;
}

esp_status esp_debug_fail_alloc(esp_ctx *ctx, int64_t n)
{
    if (!ctx)
        return ESP_ERR_INVALID_ARG;
    ctx->fail_alloc_in = n < 0 ? -1 : n;
    return ESP_OK;
}

esp_status esp_debug_set_interleave(esp_ctx *ctx, int32_t enable)
{
    esp_status st = check_ctx(ctx);
    if (st != ESP_OK)
        return st;
    ctx->il_enabled = enable != 0;
    return ESP_OK;
}

esp_status esp_debug_pass_kernel(esp_ctx *ctx, int32_t *kind)
{
    esp_status st = check_ctx(ctx);
    if (st != ESP_OK)
        return st;
    if (!kind)
        return ESP_ERR_INVALID_ARG;
    if (!ctx->loaded)
        return ESP_ERR_NOT_LOADED;
    *kind = ctx->placement ? 2 : ctx->il ? (ctx->il_f32 ? 3 : 1) : 0;
    return ESP_OK;
}

esp_status esp_debug_set_persistent(esp_ctx *ctx, int32_t mode)
{
    esp_status st = check_ctx(ctx);
    if (st != ESP_OK)
        return st;
    if (mode < -1 || mode > 1)
        return ESP_ERR_INVALID_ARG;
    ctx->persist_mode = mode;
    return ESP_OK;
}

esp_status esp_debug_persistent(esp_ctx *ctx, int32_t *grid)
{
    esp_status st = check_ctx(ctx);
    if (st != ESP_OK)
        return st;
    if (!grid)
        return ESP_ERR_INVALID_ARG;
    if (!ctx->loaded)
        return ESP_ERR_NOT_LOADED;
    *grid = (ctx->persist_mode > 0 || (ctx->persist_mode < 0 && ctx->persist_auto)) ? ctx->persist_grid : 0;
    return ESP_OK;
}

esp_status esp_debug_set_stage_f32(esp_ctx *ctx, int32_t enable)
{
    esp_status st = check_ctx(ctx);
    if (st != ESP_OK)
        return st;
    ctx->il_f32_enabled = enable != 0;
    return ESP_OK;
}

esp_status esp_debug_hold_barrier(esp_ctx *ctx)
{
    esp_status st = check_ctx(ctx);
    if (st != ESP_OK)
        return st;
    if (!ctx->loaded || !ctx->placement || !ctx->place_res_ok)
        return ESP_ERR_UNSUPPORTED;
    ctx->hold_barrier = true;
    return ESP_OK;
}

}  // extern "C"
