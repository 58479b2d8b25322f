/*
 * Oracle for the Elastic Shadow Pricing (ESP) tatonnement of Sec. 3.2.
 *
 * TEST INFRASTRUCTURE: a plain, slow, single-threaded fp64 restatement of the method that the
 * tests, __graft_entry__.smoke() and bench.py's CPU-baseline / reference legs compare the CUDA path
 * against. The product never loads it. It shares no code with the library.
 *
 * Build: cc -O2 -ffp-contract=off -std=c11 -fPIC -shared esp_oracle.c -lm
 * -ffp-contract=off matters: every fused multiply-add below is an explicit fma(), and no other
 * expression may be contracted (GCC on aarch64 contracts a*b+c by default).
 *
 * Each round (Sec. 3.2.2-3.2.3, Alg. 1 "EspTatonnement" then the final argmin):
 *   a2  effective prices p_k from lambda_k                         (Eq. price_update, reading of units)
 *   a3  reduced cost s = -v + sum_r p_{k(o,r)} * u_{o,r}            (Eq. esp_score without Gamma;
 *                                                                    negated Eq. lagrangian term)
 *   a4  per-job argmin of s, ties to the lowest local index        (Sec. 3.2.2 per-job subproblem)
 *   a5  U_k = sum_j units of the chosen options, int64              (U_r under Eq. price_update)
 *   a6  lambda_k <- max(0, lambda_k + eta_t * (U_k - C_k))          (Eq. price_update)
 */
#include "esp_oracle.h"

#include <math.h>
#include <stdlib.h>
#include <string.h>

int32_t esp_oracle_price_index(const esp_oracle_table *t, int64_t o, int32_t r)
{
    if (t->group == NULL || r < t->r_global)
        return r;
    return t->r_global + (t->R - t->r_global) * (int32_t)t->group[o] + (r - t->r_global);
}

/* a2. RAW: p_k = lambda_k, Eq. price_update applied to the units as stored.
 * NORMALIZED: Eq. price_update applied to capacity fractions u/C_k (capacity 1); a lambda on that
 * scale costs lambda_k / C_k per stored unit. */
void esp_oracle_effective_prices(const esp_oracle_table *t, int32_t s, int32_t mode,
                                 const double *lambda, double *p)
{
    const int64_t *cap = t->capacity + (int64_t)s * t->P;
    for (int32_t k = 0; k < t->P; ++k) {
        if (mode == ESP_ORACLE_NORMALIZED)
            p[k] = lambda[k] / (double)cap[k];
        else
            p[k] = lambda[k];
    }
}

/* a3. Start from -v and add the rent of each stored column in the order r = 0 .. R-1, one correctly
 * rounded fused multiply-add per column. */
double esp_oracle_reduced_cost(const esp_oracle_table *t, int64_t o, const double *p)
{
    double score = -t->values[o];
    for (int32_t r = 0; r < t->R; ++r) {
        double price = p[esp_oracle_price_index(t, o, r)];
        double amount = (double)t->units[o * t->R + r];
        score = fma(price, amount, score);
    }
    return score;
}

/* a3 + a4 + a5 for every job of scenario s. */
void esp_oracle_best_response(const esp_oracle_table *t, int32_t s, int32_t mode,
                              const double *lambda, int32_t *sel, int64_t *demand,
                              double *min_score)
{
    double *p = (double *)malloc(sizeof(double) * (size_t)t->P);
    esp_oracle_effective_prices(t, s, mode, lambda, p);
    for (int32_t k = 0; k < t->P; ++k)
        demand[k] = 0;

    for (int32_t j = 0; j < t->J; ++j) {
        int64_t first = t->job_off[(int64_t)s * t->J + j];
        int64_t last = t->job_off[(int64_t)s * t->J + j + 1];
        int64_t best = first;
        double best_score = esp_oracle_reduced_cost(t, first, p);
        for (int64_t o = first + 1; o < last; ++o) {
            double score = esp_oracle_reduced_cost(t, o, p);
            if (score < best_score) { /* strict: an equal score keeps the lower index */
                best_score = score;
                best = o;
            }
        }
        sel[j] = (int32_t)(best - first);
        if (min_score)
            min_score[j] = best_score;
        for (int32_t r = 0; r < t->R; ++r)
            demand[esp_oracle_price_index(t, best, r)] += (int64_t)t->units[best * t->R + r];
    }
    free(p);
}

/* g(lambda) = sum_j max_c [v - rent] + sum_k lambda_k C_k (Eq. lagrangian at the maximising x).
 * NORMALIZED prices live on capacity fractions, whose capacity is 1. */
double esp_oracle_dual_value(const esp_oracle_table *t, int32_t s, int32_t mode,
                             const double *lambda, const double *min_score)
{
    const int64_t *cap = t->capacity + (int64_t)s * t->P;
    double g = 0.0;
    for (int32_t j = 0; j < t->J; ++j)
        g += -min_score[j];
    for (int32_t k = 0; k < t->P; ++k) {
        if (mode == ESP_ORACLE_NORMALIZED)
            g += lambda[k];
        else
            g += lambda[k] * (double)cap[k];
    }
    return g;
}

/* a6. eta_t = eta0 (fixed) or eta0 / sqrt(t) with t the 1-based update number (Sec. 3.2.3).
 * The excess U_k - C_k is exact in int64 and converted once; in NORMALIZED mode it is divided by C_k. */
int esp_oracle_price_update(const esp_oracle_table *t, int32_t s, const esp_oracle_params *prm,
                            int32_t t1, const int64_t *demand, const double *lambda_in,
                            double *lambda_out)
{
    const int64_t *cap = t->capacity + (int64_t)s * t->P;
    double eta = prm->eta0;
    if (prm->step == ESP_ORACLE_STEP_INV_SQRT)
        eta = prm->eta0 / sqrt((double)t1);
    int status = 0;
    for (int32_t k = 0; k < t->P; ++k) {
        double excess = (double)(demand[k] - cap[k]);
        if (prm->mode == ESP_ORACLE_NORMALIZED)
            excess = excess / (double)cap[k];
        double moved = fma(eta, excess, lambda_in[k]);
        lambda_out[k] = moved > 0.0 ? moved : 0.0; /* projection onto lambda >= 0 */
        if (!isfinite(lambda_out[k]))
            status = 2;
    }
    return status;
}

static uint64_t splitmix64_mix(uint64_t z)
{
    z = (z ^ (z >> 30)) * 0xbf58476d1ce4e5b9ULL;
    z = (z ^ (z >> 27)) * 0x94d049bb133111ebULL;
    return z ^ (z >> 31);
}

uint64_t esp_oracle_selection_hash(int32_t J, const int32_t *sel)
{
    uint64_t h = 0;
    for (int32_t j = 0; j < J; ++j)
        h += splitmix64_mix(((uint64_t)(uint32_t)j << 32) | (uint64_t)(uint32_t)sel[j]);
    return h;
}

int esp_oracle_solve(const esp_oracle_table *t, int32_t s, const esp_oracle_params *prm,
                     const double *lambda0, double *lambda_out, int32_t *sel_out,
                     int64_t *demand_out, double *min_score_out, esp_oracle_result *res,
                     double *lambda_trace, int64_t *demand_trace, uint64_t *selhash_trace,
                     double *dual_trace, int32_t *sel_trace)
{
    const int32_t P = t->P, J = t->J, T = prm->max_rounds;
    double *lambda = (double *)calloc((size_t)P, sizeof(double));
    double *next = (double *)calloc((size_t)P, sizeof(double));
    int64_t *demand = (int64_t *)calloc((size_t)P, sizeof(int64_t));
    int32_t *sel = (int32_t *)calloc((size_t)(J > 0 ? J : 1), sizeof(int32_t));
    double *score = (double *)calloc((size_t)(J > 0 ? J : 1), sizeof(double));
    if (lambda0)
        memcpy(lambda, lambda0, sizeof(double) * (size_t)P);

    int status = 0, converged = 0, rounds = 0;
    double best_dual = INFINITY;
    for (int32_t it = 0; it < T; ++it) {
        if (lambda_trace)
            memcpy(lambda_trace + (int64_t)it * P, lambda, sizeof(double) * (size_t)P);
        esp_oracle_best_response(t, s, prm->mode, lambda, sel, demand, score);
        double g = esp_oracle_dual_value(t, s, prm->mode, lambda, score);
        if (g < best_dual)
            best_dual = g;
        if (dual_trace)
            dual_trace[it] = g;
        if (demand_trace)
            memcpy(demand_trace + (int64_t)it * P, demand, sizeof(int64_t) * (size_t)P);
        if (selhash_trace)
            selhash_trace[it] = esp_oracle_selection_hash(J, sel);
        if (sel_trace)
            memcpy(sel_trace + (int64_t)it * J, sel, sizeof(int32_t) * (size_t)J);

        status = esp_oracle_price_update(t, s, prm, it + 1, demand, lambda, next);
        if (status != 0)
            break;
        rounds = it + 1;

        if (prm->tol > 0.0) {
            /* Sec. 3.2.2 stops "until the prices converge" without a rule; this one stops when no
             * price moved by more than tol relative to max(1, largest price). */
            double delta = 0.0, scale = 1.0;
            for (int32_t k = 0; k < P; ++k) {
                double d = fabs(next[k] - lambda[k]);
                if (d > delta)
                    delta = d;
                if (fabs(lambda[k]) > scale)
                    scale = fabs(lambda[k]);
            }
            converged = delta <= prm->tol * scale;
        }
        memcpy(lambda, next, sizeof(double) * (size_t)P);
        if (converged)
            break;
    }

    /* Final argmin at the last prices, with no further update (Alg. 1, the loop after EspTatonnement). */
    if (lambda_trace)
        memcpy(lambda_trace + (int64_t)rounds * P, lambda, sizeof(double) * (size_t)P);
    esp_oracle_best_response(t, s, prm->mode, lambda, sel, demand, score);
    double g = esp_oracle_dual_value(t, s, prm->mode, lambda, score);
    if (g < best_dual)
        best_dual = g;
    if (dual_trace)
        dual_trace[rounds] = g;

    const int64_t *cap = t->capacity + (int64_t)s * P;
    double primal = 0.0;
    int feasible = 1;
    for (int32_t j = 0; j < J; ++j)
        primal += t->values[t->job_off[(int64_t)s * J + j] + sel[j]];
    for (int32_t k = 0; k < P; ++k)
        if (demand[k] > cap[k])
            feasible = 0;

    memcpy(lambda_out, lambda, sizeof(double) * (size_t)P);
    memcpy(sel_out, sel, sizeof(int32_t) * (size_t)J);
    memcpy(demand_out, demand, sizeof(int64_t) * (size_t)P);
    if (min_score_out)
        memcpy(min_score_out, score, sizeof(double) * (size_t)J);
    res->rounds_run = rounds;
    res->converged = converged;
    res->feasible = feasible;
    res->status = status;
    res->primal = primal;
    res->dual = g;
    res->best_dual = best_dual;

    free(lambda);
    free(next);
    free(demand);
    free(sel);
    free(score);
    return status;
}

/* Eq. adaptive_threshold (Sec. 3.3, interference-aware co-location). */
double esp_oracle_adaptive_threshold(double tau_base, double beta, double util, double util_target,
                                     double beta_max)
{
    double add = beta * (util / util_target - 1.0);
    if (add > beta_max)
        add = beta_max;
    return tau_base + add;
}

/* Gamma of Eq. esp_score (Sec. 3.2.3): switching cost and interference penalty. */
double esp_oracle_penalty(int32_t c, int32_t c_cur, double gamma0, double alpha, double s_hat, double tau)
{
    const double sw = (c_cur >= 0 && c != c_cur) ? gamma0 : 0.0;
    double excess = s_hat - tau;
    if (excess < 0.0)
        excess = 0.0;
    const double interference = alpha * excess;
    return sw + interference;
}

void esp_oracle_penalized_values(const esp_oracle_table *t, double gamma0, const int32_t *c_cur, double alpha,
                                 const double *s_hat, const double *tau, double *values_out)
{
    const int64_t n_jobs = (int64_t)t->S * t->J;
    for (int64_t j = 0; j < n_jobs; ++j) {
        const int32_t cur = c_cur ? c_cur[j] : -1;
        for (int64_t o = t->job_off[j]; o < t->job_off[j + 1]; ++o) {
            const int32_t c = (int32_t)(o - t->job_off[j]);
            const double gamma = esp_oracle_penalty(c, cur, gamma0, s_hat ? alpha : 0.0, s_hat ? s_hat[o] : 0.0,
                                                    s_hat ? tau[j] : 0.0);
            values_out[o] = t->values[o] - gamma;
        }
    }
}

/* Eq. effective_capacity (Sec. 3.4, queue-aware capacity reservation). */
void esp_oracle_effective_capacity(int32_t R, const int64_t *capacity, int32_t Q, const int64_t *q_off,
                                   const int32_t *q_units, double gamma, int64_t *c_eff)
{
    for (int32_t r = 0; r < R; ++r) {
        int64_t reserved = 0;
        for (int32_t q = 0; q < Q; ++q) {
            int32_t m = q_units[q_off[q] * R + r];
            for (int64_t o = q_off[q] + 1; o < q_off[q + 1]; ++o)
                if (q_units[o * R + r] < m)
                    m = q_units[o * R + r];
            reserved += m;
        }
        const double left = (double)capacity[r] - gamma * (double)reserved;
        int64_t c = (int64_t)floor(left);
        if (c < 1)
            c = 1;
        c_eff[r] = c;
    }
}
