/*
 * esp.h - C ABI of the GB300 (sm_103a) Elastic Shadow Pricing solver.
 *
 * The solver runs the tatonnement of Sec. 3.2 of the paper ("Elastic Shadow Pricing") on one GPU:
 * every round each job evaluates all of its configurations at the current shadow prices and keeps
 * the cheapest (Sec. 3.2.2, the per-job subproblem of Eq. lagrangian; Eq. esp_score without the
 * Gamma term), the chosen demands are summed per resource in int64 (U_r of Eq. price_update), and
 * the prices take the projected-subgradient step of Eq. price_update. After the last update one
 * more best response at the final prices gives the returned selection (Alg. 1, the argmin that
 * follows EspTatonnement). S independent problems ("scenarios") are solved in one call.
 *
 * Conventions
 *  - Every function returns an esp_status; no exception or longjmp crosses this boundary.
 *  - Pointers documented as "host" are ordinary host memory owned by the caller; inputs are copied
 *    during the call, outputs are written before it returns. Pinned host memory makes copies faster
 *    but is not required. Pointers documented as "device" are CUDA device pointers on the context's
 *    device, owned by the caller.
 *  - A context is used by one host thread at a time. All GPU work of a context runs on its stream.
 *  - After ESP_ERR_CUDA or ESP_ERR_TIMEOUT the context refuses further work with ESP_ERR_STATE;
 *    only esp_destroy is valid then.
 *  - The integer program's performance floor (Eq. perf_constraint: T_j(c) >= L_j) is the caller's
 *    job: pass only the configurations that meet it, with value v = w_j * T_j(c) (Eq. primal_obj).
 */
#ifndef ESP_H
#define ESP_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define ESP_ABI_VERSION 1

typedef struct esp_ctx esp_ctx;

typedef enum {
    ESP_OK = 0,
    ESP_ERR_INVALID_ARG = 1, /* bad pointer, size or table content (see esp_load_options) */
    ESP_ERR_OVERFLOW = 2,    /* a demand total could leave int64, or a price became non-finite */
    ESP_ERR_OOM = 3,         /* device or host allocation failed */
    ESP_ERR_CUDA = 4,        /* a CUDA call failed; the context is unusable afterwards */
    ESP_ERR_NOT_LOADED = 5,  /* esp_solve / esp_evaluate / getters before a table was loaded or solved */
    ESP_ERR_TIMEOUT = 6,     /* a bounded device wait gave up; the context is unusable afterwards */
    ESP_ERR_STATE = 7,       /* the context was poisoned by an earlier ESP_ERR_CUDA / ESP_ERR_TIMEOUT */
    ESP_ERR_UNSUPPORTED = 8  /* no GPU, or the device is not sm_103 */
} esp_status;

/* Units of lambda (the paper leaves them open; Sec. 3.2.3).
 * RAW: Eq. price_update verbatim on the stored units: lambda_k += eta_t * (U_k - C_k); a unit of
 *      resource k costs lambda_k.
 * NORMALIZED: the same equation on capacity fractions u / C_k (capacity 1):
 *      lambda_k += eta_t * (U_k - C_k) / C_k; a stored unit of resource k costs lambda_k / C_k. */
typedef enum { ESP_PRICE_RAW = 0, ESP_PRICE_NORMALIZED = 1 } esp_price_mode;

/* eta_t of Eq. price_update: fixed eta0, or eta0 / sqrt(t) with t = 1 for the first update. */
typedef enum { ESP_STEP_FIXED = 0, ESP_STEP_INV_SQRT = 1 } esp_step_rule;

/* esp_params.flags */
#define ESP_FLAG_EXACT_ONLY 0x1u       /* evaluate every option in fp64 (no fp32 screen); same results, slower */
#define ESP_FLAG_PER_ROUND_LAUNCH 0x2u /* price update as its own launch after every evaluation pass, instead of
                                          by the pass's last warp per scenario (same results) */
#define ESP_FLAG_PASS_EVENTS 0x4u      /* record a CUDA event pair around every evaluation-pass launch (inside the
                                          solve's CUDA graph on a non-default stream); read with esp_pass_times */
#define ESP_FLAG_RESIDENT 0x8u         /* run all rounds of a scenario in one launch, its table held in the shared
                                          memory of one thread-block cluster for the whole solve (no table bytes
                                          read from HBM after the first round). Taken when the table has no group
                                          column, each scenario fits in a cluster (up to 16 CTAs of up to about
                                          227 KB) and the library's cost model predicts it faster than streaming
                                          (a batch of many scenarios needs many waves of clusters and usually is
                                          not); otherwise the streaming path runs. Same results either way.
                                          esp_last_launch_count tells which ran (3: resident); with
                                          ESP_FLAG_PASS_EVENTS the one resident launch counts as one pass.
                                          For a table loaded with esp_load_placement it selects the
                                          grid-resident solve instead: all rounds in one cooperative launch
                                          with a grid-wide barrier per round (4 launches; S*P <= 4096, no
                                          fingerprint or dual trace; otherwise per-round launches) */

typedef struct {
    double eta0;            /* > 0, finite */
    int32_t step;           /* esp_step_rule */
    int32_t mode;           /* esp_price_mode */
    int32_t max_rounds;     /* T >= 0: number of price updates (fewer if tol stops a scenario) */
    uint32_t flags;         /* ESP_FLAG_* */
    double tol;             /* >= 0. 0: exactly T updates. > 0: a scenario stops after the update in
                               which max_k |lambda'_k - lambda_k| <= tol * max(1, max_k |lambda_k|) */
    const double *lambda0;  /* host, S*P initial prices (>= 0, finite), or NULL for zeros. Warm start
                               (Sec. 3.4, "warm starting") and resume both pass saved prices here. */
    /* Optional host trace buffers, NULL to skip (tracing makes the solve slower). Layout is
     * scenario-major. Rows of rounds a scenario did not run are left as they were. */
    double *lambda_trace;   /* S*(T+1)*P: row t = lambda^t, the prices evaluated in round t */
    int64_t *demand_trace;  /* S*T*P: U^t, the demand of round t's selection */
    uint64_t *selhash_trace;/* S*T: sum over jobs j of splitmix64_mix((j << 32) | c_j) of round t */
    double *dual_trace;     /* S*(T+1): g(lambda^t) of Eq. lagrangian; entry rounds_run is the final one */
    uint64_t *round_time_trace; /* S*T: the GPU's global timer (ns) when round t's price update of the
                               scenario was applied (on every solve path); differences of consecutive
                               entries are the scenario's round times */
} esp_params;

typedef struct {
    int32_t rounds_run;     /* price updates performed */
    int32_t converged;      /* 1 if tol > 0 stopped this scenario */
    int32_t feasible;       /* 1 if the final demand is <= capacity in every priced resource */
    int32_t status;         /* ESP_OK, or ESP_ERR_OVERFLOW if a price became non-finite (the scenario
                               then stops at its last finite prices) */
    double primal;          /* sum_j v(c_j*) at the final selection (Eq. primal_obj) */
    double dual;            /* g(lambda) at the final prices (Eq. lagrangian maximised over x) */
    double best_dual;       /* min over evaluated rounds of g(lambda^t) when dual_trace is given,
                               else equal to dual */
    float device_ms;        /* device time of the whole solve (every launch of it, all scenarios),
                               from a CUDA event pair around it on the context's stream */
} esp_result;

/* Creates a context on `device` (-1: the current device) that issues all work on `cuda_stream`
 * (a cudaStream_t; NULL: the legacy default stream). *out receives the context.
 * Errors: ESP_ERR_INVALID_ARG (out NULL), ESP_ERR_UNSUPPORTED (no device or not sm_103),
 * ESP_ERR_CUDA, ESP_ERR_OOM. */
esp_status esp_create(esp_ctx **out, int device, void *cuda_stream);

/* Changes the stream later work is issued on (e.g. to follow a framework's current stream). */
esp_status esp_set_stream(esp_ctx *ctx, void *cuda_stream);

/* Loads the option table (Sec. 3.1's profiles, the data of the integer program of Sec. 3.2.1):
 * S scenarios of J jobs each; job j of scenario s owns global options
 * job_offsets[s*J + j] .. job_offsets[s*J + j + 1] - 1 (job-major, options of a job contiguous).
 *   job_offsets  host, S*J + 1 int64: job_offsets[0] = 0, every job has >= 1 option
 *   units        host, n_opt*R int32 >= 0, row-major: units[o*R + r] = R_j(c)[r] of option o
 *   values       host, n_opt fp64, finite: w_j*T_j(c), larger is better
 *   group        host, n_opt uint16 or NULL. NULL: P == R == r_global and column r is priced by
 *                lambda_r. Else: columns r < r_global are priced globally, column r >= r_global of
 *                option o by lambda[r_global + (R - r_global)*group[o] + (r - r_global)], and
 *                P == r_global + (R - r_global) * n_groups with group[o] < n_groups.
 *   capacity     host, S*P int64 > 0: C_k of scenario s at [s*P + k]
 * 1 <= R <= 16, 0 <= r_global <= R, 1 <= P, S >= 1, J >= 0; no job may hold more than 2^31 - 1
 * options and J*R < 2^32 (every demand total then fits in int64).
 * The table is copied into device memory owned by the context; a previous table is released.
 * Content is validated on the device; errors: ESP_ERR_INVALID_ARG (shape or content),
 * ESP_ERR_OOM, ESP_ERR_CUDA. */
esp_status esp_load_options(esp_ctx *ctx, int32_t S, int32_t J, int32_t R, int32_t P, int32_t r_global,
                            const int64_t *job_offsets, const int32_t *units, const double *values,
                            const uint16_t *group, const int64_t *capacity);

/* As esp_load_options with every table pointer a device pointer (e.g. a framework tensor's data);
 * the data is copied device-to-device on the context's stream. */
esp_status esp_load_options_device(esp_ctx *ctx, int32_t S, int32_t J, int32_t R, int32_t P,
                                   int32_t r_global, const int64_t *job_offsets, const int32_t *units,
                                   const double *values, const uint16_t *group,
                                   const int64_t *capacity);

/* Runs the tatonnement of every scenario (Sec. 3.2.3, Eq. price_update; Alg. 1's EspTatonnement
 * followed by the final argmin) and, if `out` is not NULL, writes S esp_result entries (host).
 * Blocks until the GPU finishes. Errors: ESP_ERR_NOT_LOADED, ESP_ERR_INVALID_ARG (params),
 * ESP_ERR_OVERFLOW (some scenario's prices became non-finite; results are still written),
 * ESP_ERR_TIMEOUT, ESP_ERR_CUDA. */
esp_status esp_solve(esp_ctx *ctx, const esp_params *params, esp_result *out);

/* As esp_solve without blocking and without host traces (the trace pointers must be NULL): the work
 * is queued on the context's stream. Call esp_get_result / the getters afterwards (they wait).
 * lambda0, when given, is read before the call returns. */
esp_status esp_solve_async(esp_ctx *ctx, const esp_params *params);

/* Results of the last solve (host outputs; each call waits for the context's stream). */
esp_status esp_get_result(esp_ctx *ctx, esp_result *out);       /* S entries */
esp_status esp_get_prices(esp_ctx *ctx, double *out);            /* S*P final lambda */
esp_status esp_get_selection(esp_ctx *ctx, int32_t *out);        /* S*J local option index 0..K_j-1 */
esp_status esp_get_demand(esp_ctx *ctx, int64_t *out);           /* S*P demand of the final selection */

/* One best response (Sec. 3.2.2's per-job argmax, ties to the lowest local index) at caller prices,
 * without any price update. lambda: host S*P (>= 0, finite) in the units of `mode`. Outputs (host,
 * each may be NULL): sel S*J, demand S*P, min_score S*J (each job's smallest reduced cost
 * rent - value, fp64). Blocks. Errors: ESP_ERR_NOT_LOADED, ESP_ERR_INVALID_ARG, ESP_ERR_CUDA. */
esp_status esp_evaluate(esp_ctx *ctx, const double *lambda, int32_t mode, uint32_t flags, int32_t *sel,
                        int64_t *demand, double *min_score);

/* Best response at caller prices that allocates nothing (no cudaMalloc, no cudaFree, no host or
 * device allocation by the library). The paper has no counterpart: this exists for callers that
 * cannot allocate device memory where they need the answer, e.g. code running while another
 * framework's caching allocator owns the device, or a scheduler loop that must not stall on the
 * device synchronisation that cudaMalloc / cudaFree imply and works from memory reserved up front.
 * Every pointer is a device pointer owned by the caller: the table (job_offsets S*J+1 int64,
 * units n_opt*R int32 >= 0, values n_opt fp64 finite; R <= 16, no groups; a job with no options
 * gets sel = -1, min_score = +inf and adds no demand),
 * capacity S*R int64 > 0, lambda S*R (>= 0, finite, in the units of `mode`), and the outputs sel
 * S*J, demand S*R (overwritten; int64), min_score S*J (may be NULL). The inputs are not validated.
 * The per-unit prices go to one fixed scratch array of 65536 fp64 in the library's device memory,
 * so S*R must not exceed 65536 (ESP_ERR_INVALID_ARG otherwise). The array exists once per GPU, is
 * shared by every call and keeps the last call's contents; calls that may overlap on the GPU (on
 * different streams, or from different threads) race on it and must be serialised by the caller.
 * The first call on a device looks up the array's device address (once per device, under a lock);
 * make that first call before any stream capture. The address is kept until the process exits, so
 * the entry point must not be used across a cudaDeviceReset of that device. Work is queued on `cuda_stream` (NULL: the legacy
 * default stream); the call returns without waiting. Results equal esp_evaluate's.
 * Errors: ESP_ERR_INVALID_ARG, ESP_ERR_UNSUPPORTED (device index >= 64), ESP_ERR_CUDA. */
esp_status esp_evaluate_noalloc(int32_t S, int32_t J, int32_t R, const int64_t *job_offsets, const int32_t *units,
                                const double *values, const int64_t *capacity, const double *lambda, int32_t mode,
                                int32_t *sel, int64_t *demand, double *min_score, void *cuda_stream);

/* Loads a placement-expanded table in factored form (Sec. 3.3: configurations crossed with nodes,
 * the co-location slowdown folded into the value), replacing any loaded table. Job j of scenario s
 * (global job index s*J + j) has KC configurations and KC * N options; option (k, n) has local index
 * k * N + n, the units of configuration k — columns r < r_global priced by lambda_r, columns
 * r >= r_global by lambda[r_global + (R - r_global)*n + (r - r_global)], so P = r_global +
 * (R - r_global) * N — and the value
 *     cfg_values[j*KC + k] - (double)(sens[j] * D[job_type[j]*NT + node_type[n]])
 * with the product taken in fp32. The solve is the one esp_load_options would give for the
 * expanded table (same selections, demands, prices, objectives), computed from the factors:
 *   cfg_units   host, S*J*KC*R int32 >= 0      cfg_values host, S*J*KC fp64, finite
 *   sens        host, S*J fp32, finite           job_type   host, S*J int32 in [0, NT)
 *   node_type   host, N int32 in [0, NT)          D          host, NT*NT fp32, finite
 *   capacity    host, S*P int64 > 0
 * 1 <= KC <= 32, 1 <= N <= 64, 1 <= NT <= 64, 1 <= R <= 16, 0 <= r_global < R. esp_set_penalties
 * does not apply (ESP_ERR_UNSUPPORTED); ESP_FLAG_RESIDENT selects the grid-resident solve (see the
 * flag). Errors:
 * ESP_ERR_INVALID_ARG, ESP_ERR_UNSUPPORTED (shape beyond the limits of the device), ESP_ERR_OOM,
 * ESP_ERR_CUDA. */
esp_status esp_load_placement(esp_ctx *ctx, int32_t S, int32_t J, int32_t KC, int32_t N, int32_t R, int32_t r_global,
                              const int32_t *cfg_units, const double *cfg_values, const float *sens,
                              const int32_t *job_type, int32_t NT, const int32_t *node_type, const float *D,
                              const int64_t *capacity);

/* The Gamma term of Eq. esp_score for later solves and evaluations. Option c of job j then scores
 *     rent - v + Gamma_j(c),   Gamma_j(c) = gamma0 * [c != c_cur[j]] + alpha * max(0, s_hat[o] - tau[j]),
 * the switching cost from the job's current configuration plus the interference penalty of the
 * predicted co-location slowdown above the job's tolerance (Sec. 3.2.3 and Sec. 3.3; Alg. 1 updates
 * the slowdowns between ESP rounds). Gamma is computed in fp64 as (c != c_cur ? gamma0 : 0) +
 * alpha * max(0, s_hat - tau) and applied as the effective value v' = v - Gamma, one correctly
 * rounded operation per step; every output and objective (primal = sum of v') then refers to v'.
 *   gamma0  >= 0, finite: switching cost
 *   c_cur   host, S*J int32: current configuration of each job (local index), -1 for a job without
 *           one; NULL: no switching cost
 *   alpha   >= 0, finite: weight of the interference penalty
 *   s_hat   host, n_opt fp64: predicted slowdown of each option (IAC's output, Eq. dnn_pred); NULL:
 *           no interference penalty
 *   tau     host, S*J fp64: tolerance thresholds tau_j(t) (esp_adaptive_threshold); required with
 *           s_hat, ignored without
 * gamma0 = 0 with s_hat = NULL restores the loaded values. Errors: ESP_ERR_NOT_LOADED,
 * ESP_ERR_INVALID_ARG (bad weights, a c_cur at or beyond its job's option count, a non-finite
 * effective value; the context then holds the loaded values, without penalties). */
esp_status esp_set_penalties(esp_ctx *ctx, double gamma0, const int32_t *c_cur, double alpha, const double *s_hat,
                             const double *tau);

/* tau_j(t) of Eq. adaptive_threshold for n jobs (host only, no context):
 *     tau_out[j] = tau_base[j] + min(beta * (util / util_target - 1), beta_max),
 * util = U(t) the cluster utilization, util_target = U_target > 0; the additive term is clamped from
 * above only (Sec. 3.3). Errors: ESP_ERR_INVALID_ARG for null pointers, n < 0 or util_target <= 0. */
esp_status esp_adaptive_threshold(int64_t n, const double *tau_base, double beta, double util, double util_target,
                                  double beta_max, double *tau_out);

/* Effective capacity of Eq. effective_capacity (host only): for each of R resources
 *     c_eff[r] = floor(capacity[r] - gamma * sum over queued jobs q of min over q's options of units[o*R + r]),
 * at least 1 (a capacity must stay positive). capacity[r] lies in [1, 2^53] (exact in fp64). The queue
 * is a CSR table of Q jobs: q_offsets (Q + 1, q_offsets[0] = 0, every job >= 1 option) and q_units
 * (rows of R int32 >= 0). gamma in [0, 1] reserves capacity for the queued jobs at their componentwise
 * smallest footprint (Sec. 3.4). Errors: ESP_ERR_INVALID_ARG (also for a capacity outside that range
 * or a negative unit). */
esp_status esp_effective_capacity(int32_t R, const int64_t *capacity, int32_t Q, const int64_t *q_offsets,
                                  const int32_t *q_units, double gamma, int64_t *c_eff);

/* Number of kernel launches the last esp_solve / esp_solve_async issued. */
esp_status esp_last_launch_count(esp_ctx *ctx, int64_t *out);

/* Device time of the evaluation passes recorded with ESP_FLAG_PASS_EVENTS since the last reset:
 * *total_ms receives the summed CUDA-event durations (measured on the context's stream) and *count
 * the number of passes. Solves on the legacy default stream contribute every pass; solves replayed
 * from a CUDA graph contribute the passes of the latest replay. Waits for the stream. reset != 0
 * clears the record afterwards. */
esp_status esp_pass_times(esp_ctx *ctx, double *total_ms, int64_t *count, int32_t reset);

/* Static description of a string for a status. Never NULL. */
const char *esp_status_string(esp_status status);

/* Releases every resource of the context (NULL is allowed). */
void esp_destroy(esp_ctx *ctx);

#ifdef __cplusplus
}
#endif
#endif /* ESP_H */
