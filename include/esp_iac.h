/*
 * esp_iac.h - C ABI of the IAC slowdown predictor (Sec. 3.3 of the paper, "Interference-Aware
 * Co-location") on one GB300 (sm_103a): batched inference of the three-layer network of
 * Sec. 3.3.2 over co-location pairs, producing the predicted slowdowns S_hat that feed the
 * interference penalty of Eq. esp_score (esp_set_penalties in esp.h).
 *
 * Per-job features (Sec. 3.3.1), 14 fp32 per row, in this order:
 *    0 SM Active (fraction of cycles)   1 SM Occupancy   2 DRAM Active   3 Framebuffer Used (MB)
 *    4 Tensor Core Active   5 workload type (0 training, 1 inference)   6 log-scaled parameter count
 *    7 isolated throughput T_j(c)   8 micro-batch size   9 activation checkpointing flag
 *   10 mixed-precision flag   11 input sequence length   12 average output sequence length
 *   13 prefix caching ratio
 * (a training job's inference slots and an inference job's training slots hold 0). A row describes
 * one job in one configuration; the same job in several configurations takes several rows.
 *
 * Pair (i, j) asks for the slowdown of row i when co-located with row j. Its 36 inputs are row i,
 * row j and 8 pairwise features: the means over both rows of SM Active, SM Occupancy, DRAM Active
 * and Tensor Core Active; type_i + type_j (0 training-training, 1 mixed, 2 inference-inference);
 * the memory pressure (fb_i + fb_j) / c_mem; the compute balance min(sm_i, sm_j) / max(sm_i, sm_j)
 * (1 when both are 0); the memory intensity difference |dram_i / sm_i - dram_j / sm_j| (a term
 * whose SM Active is 0 counts as 0).
 *
 * Network (inference: dropout off, Batch Normalization with its running statistics):
 *     h1 = ReLU(BN1(W1 x + b1)),  h2 = ReLU(BN2(W2 h1 + b2)),  S_hat = 1 + ReLU(W3 h2 + b3)
 * (Eq. dnn_pred), BN(z) = gamma (z - mean) / sqrt(var + eps) + beta per unit. Each BN is folded
 * into the preceding layer when the model is loaded; the kernels compute in fp32 (the hidden layers
 * on the tensor cores with a three-term tf32 split, or as fused multiply-adds; see
 * esp_iac_set_path).
 *
 * Conventions are those of esp.h: every function returns an esp_status, "host" pointers are copied
 * during the call, "device" pointers are CUDA device pointers owned by the caller, a handle is used
 * by one host thread at a time and all its GPU work runs on its stream.
 */
#ifndef ESP_IAC_H
#define ESP_IAC_H

#include <stdint.h>

#include "esp.h"

#ifdef __cplusplus
extern "C" {
#endif

#define ESP_IAC_FEATURES 14   /* per-job row */
#define ESP_IAC_INPUTS 36     /* network input: 2 rows + 8 pairwise */
#define ESP_IAC_MAX_HIDDEN 64

typedef struct esp_iac esp_iac;

/* Kernels of esp_iac_predict (esp_iac_set_path):
 * ESP_IAC_PATH_TENSOR (default): the two hidden layers as tcgen05 tensor-core MMAs (kind::tf32,
 *     fp32 accumulators in tensor memory) on a three-term split of every operand, a = a_hi + a_lo
 *     with a_hi = a truncated to tf32 and a_lo = tf32(a - a_hi): a_hi b_hi + a_hi b_lo + a_lo b_hi,
 *     which keeps each product within 2^-19 relative of the fp32 product; biases, ReLU and the
 *     output layer on the CUDA cores.
 * ESP_IAC_PATH_FMA: everything as fp32 fused multiply-adds on the CUDA cores. */
#define ESP_IAC_PATH_TENSOR 0
#define ESP_IAC_PATH_FMA 1

/* Creates a predictor on `device` (-1: the current device) whose work runs on `cuda_stream`
 * (NULL: the legacy default stream). Errors: ESP_ERR_INVALID_ARG, ESP_ERR_UNSUPPORTED (no GPU, or
 * not sm_103), ESP_ERR_OOM, ESP_ERR_CUDA. */
esp_status esp_iac_create(esp_iac **out, int device, void *cuda_stream);

esp_status esp_iac_set_stream(esp_iac *m, void *cuda_stream);

/* Loads the network's parameters (host, fp32, row-major), replacing any earlier model:
 *   W1 H*36, b1 H, bn1 4*H (gamma, beta, running mean, running variance of BN1, each H long),
 *   W2 H*H,  b2 H, bn2 4*H,  W3 H,  b3,  eps (of both BN layers).
 * 1 <= H <= 64. Folding: s = gamma / sqrt(var + eps), W' = s W (per output row) and
 * b' = s (b - mean) + beta are computed in fp64 and rounded once to fp32. Errors:
 * ESP_ERR_INVALID_ARG (null pointer, H out of range, a non-finite parameter, eps < 0, var + eps <= 0,
 * or a folded parameter beyond fp32). */
esp_status esp_iac_load_model(esp_iac *m, int32_t H, const float *W1, const float *b1, const float *bn1,
                              const float *W2, const float *b2, const float *bn2, const float *W3, float b3,
                              float eps);

/* S_hat of every pair (device pointers, queued on the handle's stream; returns without waiting):
 *   job_features  device, n_rows * 14 fp32, finite, 8-byte aligned
 *   pairs         device, n_pairs * 2 int32 (i, j) row indices, 8-byte aligned
 *   c_mem         total GPU memory in the framebuffer's unit (MB), > 0
 *   s_hat         device, n_pairs fp32 (written)
 * A pair with an index outside [0, n_rows) gets NaN; nothing is read for it. n_pairs = 0 does
 * nothing. Errors: ESP_ERR_NOT_LOADED (no model), ESP_ERR_INVALID_ARG, ESP_ERR_CUDA. */
esp_status esp_iac_predict(esp_iac *m, int32_t n_rows, const float *job_features, int64_t n_pairs,
                           const int32_t *pairs, float c_mem, float *s_hat);

/* The same with host pointers: inputs are copied to device buffers owned by the handle (grown as
 * needed), the result is copied back, and the call waits for it. Pair indices are checked on the
 * host (ESP_ERR_INVALID_ARG for one outside [0, n_rows)). */
esp_status esp_iac_predict_host(esp_iac *m, int32_t n_rows, const float *job_features, int64_t n_pairs,
                                const int32_t *pairs, float c_mem, float *s_hat);

/* Selects the kernel of later predictions (ESP_IAC_PATH_TENSOR or ESP_IAC_PATH_FMA). Errors:
 * ESP_ERR_INVALID_ARG for another value. */
esp_status esp_iac_set_path(esp_iac *m, int32_t path);

/* Waits for the handle's stream and reports a device-side failure of the queued predictions:
 * ESP_ERR_TIMEOUT when a bounded wait of the tensor path gave up (the handle then refuses further
 * work with ESP_ERR_STATE), ESP_ERR_CUDA on a CUDA error. esp_iac_predict_host does this itself. */
esp_status esp_iac_synchronize(esp_iac *m);

/* Number of kernel launches of the last esp_iac_predict / esp_iac_predict_host. */
esp_status esp_iac_last_launch_count(esp_iac *m, int64_t *out);

void esp_iac_destroy(esp_iac *m);

#ifdef __cplusplus
}
#endif

#endif /* ESP_IAC_H */
