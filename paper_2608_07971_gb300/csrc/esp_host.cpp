// Host-side formulas of the scheduling loop around the tatonnement: the adaptive tolerance
// threshold (Eq. adaptive_threshold) and the queue-aware effective capacity (Eq. effective_capacity).
#include <cmath>
#include <cstdint>

#include "esp.h"

namespace {
constexpr int64_t kMaxCapacity = (int64_t)1 << 53;
}

esp_status esp_adaptive_threshold(int64_t n, const double *tau_base, double beta, double util, double util_target,
                                  double beta_max, double *tau_out)
{
    if (n < 0 || (n > 0 && (!tau_base || !tau_out)) || !(util_target > 0.0) || !std::isfinite(beta) ||
        !std::isfinite(util) || !std::isfinite(util_target) || std::isnan(beta_max))
        return ESP_ERR_INVALID_ARG;
    double add = beta * (util / util_target - 1.0);
    if (add > beta_max)
        add = beta_max;
    for (int64_t j = 0; j < n; ++j)
        tau_out[j] = tau_base[j] + add;
    return ESP_OK;
}

esp_status esp_effective_capacity(int32_t R, const int64_t *capacity, int32_t Q, const int64_t *q_offsets,
                                  const int32_t *q_units, double gamma, int64_t *c_eff)
{
    if (R < 1 || Q < 0 || !capacity || !c_eff || !q_offsets || (Q > 0 && !q_units) || !(gamma >= 0.0) ||
        !std::isfinite(gamma) || q_offsets[0] != 0)
        return ESP_ERR_INVALID_ARG;
    for (int32_t q = 0; q < Q; ++q)
        if (q_offsets[q + 1] <= q_offsets[q])
            return ESP_ERR_INVALID_ARG;
    // Capacities up to 2^53 convert to double exactly, so the floor below stays within int64.
    for (int32_t r = 0; r < R; ++r)
        if (capacity[r] < 1 || capacity[r] > kMaxCapacity)
            return ESP_ERR_INVALID_ARG;
    for (int32_t r = 0; r < R; ++r) {
        int64_t reserved = 0;
        for (int32_t q = 0; q < Q; ++q) {
            int32_t m = q_units[q_offsets[q] * R + r];
            for (int64_t o = q_offsets[q] + 1; o < q_offsets[q + 1]; ++o)
                m = q_units[o * R + r] < m ? q_units[o * R + r] : m;
            if (m < 0)
                return ESP_ERR_INVALID_ARG;
            reserved += m;
        }
        const double left = (double)capacity[r] - gamma * (double)reserved;
        const double f = std::floor(left);
        c_eff[r] = (f < 1.0) ? 1 : (int64_t)f;
    }
    return ESP_OK;
}
