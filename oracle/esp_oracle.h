/*
 * Oracle for the Elastic Shadow Pricing (ESP) tatonnement of Sec. 3.2.
 *
 * TEST INFRASTRUCTURE. This is a plain, slow, single-threaded fp64 restatement of the method,
 * used only to check the CUDA path: only tests/, __graft_entry__.smoke() and the cpu_baseline /
 * reference legs of bench.py may load it. It shares no code, header or constant with the library
 * under paper_2608_07971_gb300/ and never includes anything from there.
 *
 * Notation follows Sec. 3.2: jobs j, configuration (option) c, resource r, units R_j(c)[r],
 * value w_j*T_j(c) (stored as one fp64 number v), capacity C_r, shadow price lambda_r.
 */
#ifndef ESP_ORACLE_H
#define ESP_ORACLE_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* One batch of S independent allocation problems (scenarios), each with J jobs.
 * Options of job j of scenario s are the global option indices
 * job_off[s*J + j] .. job_off[s*J + j + 1] - 1 (CSR, job-major, configuration-contiguous).
 * units[o*R + r] is R_j(c)[r] for global option o. With group == NULL every column r is priced by
 * lambda_r (P == R). With group != NULL the first r_global columns are priced globally and column
 * r >= r_global of option o is priced by lambda[r_global + (R - r_global)*group[o] + (r - r_global)]. */
typedef struct {
    int32_t S, J, R, P, r_global;
    const int64_t *job_off;   /* S*J + 1 */
    const int32_t *units;     /* n_opt * R */
    const double *values;     /* n_opt */
    const uint16_t *group;    /* n_opt or NULL */
    const int64_t *capacity;  /* S * P */
} esp_oracle_table;

enum { ESP_ORACLE_RAW = 0, ESP_ORACLE_NORMALIZED = 1 };
enum { ESP_ORACLE_STEP_FIXED = 0, ESP_ORACLE_STEP_INV_SQRT = 1 };

typedef struct {
    double eta0;
    int32_t step;       /* ESP_ORACLE_STEP_* */
    int32_t mode;       /* ESP_ORACLE_RAW / NORMALIZED */
    int32_t max_rounds; /* T */
    double tol;         /* 0: run exactly T price updates */
} esp_oracle_params;

typedef struct {
    int32_t rounds_run;  /* price updates performed */
    int32_t converged;
    int32_t feasible;    /* final demand <= capacity in every priced resource */
    int32_t status;      /* 0 ok, 2 a price became non-finite */
    double primal;       /* sum_j v(c_j*) at the final selection */
    double dual;         /* g(lambda) at the final prices */
    double best_dual;    /* min over every evaluated round of g(lambda^t) */
} esp_oracle_result;

/* Price column of (option o, stored column r). */
int32_t esp_oracle_price_index(const esp_oracle_table *t, int64_t o, int32_t r);

/* Effective per-unit price of each priced resource (Eq. price_update's lambda in raw units, or a
 * capacity-normalised lambda divided by C_k). lambda, p: P entries of scenario s. */
void esp_oracle_effective_prices(const esp_oracle_table *t, int32_t s, int32_t mode,
                                 const double *lambda, double *p);

/* Reduced cost of option o at effective prices p: rent minus value (Eq. esp_score without the
 * Gamma term; the negated per-job Lagrangian term of Eq. lagrangian). */
double esp_oracle_reduced_cost(const esp_oracle_table *t, int64_t o, const double *p);

/* Best response of every job of scenario s at lambda (Alg. 1, argmin of Score), the aggregate demand
 * U_k of the chosen options (Eq. price_update's U_r) and each job's minimal reduced cost.
 * sel: J local indices; demand: P; min_score: J (may be NULL). */
void esp_oracle_best_response(const esp_oracle_table *t, int32_t s, int32_t mode,
                              const double *lambda, int32_t *sel, int64_t *demand,
                              double *min_score);

/* g(lambda) of Eq. lagrangian from the minimal reduced costs of a best response. */
double esp_oracle_dual_value(const esp_oracle_table *t, int32_t s, int32_t mode,
                             const double *lambda, const double *min_score);

/* One projected-subgradient step of Eq. price_update for update number t1 (1-based).
 * Returns 0, or 2 if a price became non-finite. */
int esp_oracle_price_update(const esp_oracle_table *t, int32_t s, const esp_oracle_params *prm,
                            int32_t t1, const int64_t *demand, const double *lambda_in,
                            double *lambda_out);

/* Order-independent fingerprint of a selection: sum over jobs of splitmix64_mix((j << 32) | c_j). */
uint64_t esp_oracle_selection_hash(int32_t J, const int32_t *sel);

/* The whole tatonnement of one scenario (Sec. 3.2.3, Alg. 1's EspTatonnement and the final argmin).
 * lambda0: P entries or NULL (zeros). Outputs: lambda_out (P), sel_out (J), demand_out (P, the
 * demand of the final selection), min_score_out (J, may be NULL).
 * Optional traces (NULL to skip): lambda_trace ((T+1)*P, row t = lambda^t, rows after convergence
 * repeat the frozen prices), demand_trace (T*P, U^t), selhash_trace (T), dual_trace (T+1),
 * sel_trace (T*J). Returns the status also stored in res->status. */
int esp_oracle_solve(const esp_oracle_table *t, int32_t s, const esp_oracle_params *prm,
                     const double *lambda0, double *lambda_out, int32_t *sel_out,
                     int64_t *demand_out, double *min_score_out, esp_oracle_result *res,
                     double *lambda_trace, int64_t *demand_trace, uint64_t *selhash_trace,
                     double *dual_trace, int32_t *sel_trace);

/* tau_j(t) of Eq. adaptive_threshold: tau_base + beta * (U(t) / U_target - 1), the additive term
 * clamped from above at beta_max (Sec. 3.3: tau_j(t) <= tau_base + beta_max). */
double esp_oracle_adaptive_threshold(double tau_base, double beta, double util, double util_target,
                                     double beta_max);

/* Gamma_j^(m)(c) of Eq. esp_score for option c of a job: the switching cost gamma0 * [c != c_cur]
 * (no switching cost when c_cur < 0, a job without a current configuration) plus the interference
 * penalty alpha * max(0, s_hat - tau) with s_hat the predicted co-location slowdown of the option
 * and tau the job's threshold. */
double esp_oracle_penalty(int32_t c, int32_t c_cur, double gamma0, double alpha, double s_hat, double tau);

/* Values of Eq. esp_score with the Gamma term: v'_o = v_o - Gamma_j(c) for every option of the table
 * (the score becomes rent - v' = rent - v + Gamma). c_cur: S*J current configurations (local index,
 * -1 none) or NULL (no switching cost); s_hat: n_opt predicted slowdowns or NULL (no interference
 * penalty); tau: S*J thresholds (needed with s_hat). values_out: n_opt. */
void esp_oracle_penalized_values(const esp_oracle_table *t, double gamma0, const int32_t *c_cur, double alpha,
                                 const double *s_hat, const double *tau, double *values_out);

/* Eq. effective_capacity for P = R priced columns: C_eff_r = C_r - gamma * sum over the queued jobs q
 * of min over q's options of R_q(c)[r] (componentwise minimum footprint), rounded down to an
 * integer and kept at least 1. queue: CSR offsets q_off (Q + 1) and units q_units (rows of R). */
void esp_oracle_effective_capacity(int32_t R, const int64_t *capacity, int32_t Q, const int64_t *q_off,
                                   const int32_t *q_units, double gamma, int64_t *c_eff);

#ifdef __cplusplus
}
#endif
#endif
