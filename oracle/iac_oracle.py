"""Oracle of the IAC interference predictor (Sec. 3.3): the 36-dimensional pair feature vector of
Sec. 3.3.1 and the three-layer network of Sec. 3.3.2 / Eq. dnn_pred, in numpy fp64.

TEST INFRASTRUCTURE: only tests/, __graft_entry__.smoke() and bench.py's CPU-baseline and reference
legs may import this module. It imports nothing from the library under paper_2608_07971_gb300/.

Per-job features, in this order (Sec. 3.3.1; 14 = 5 hardware + 3 common + 3 training + 3 inference):
   0 SM Active        1 SM Occupancy     2 DRAM Active      3 Framebuffer Used (MB)   4 Tensor Core Active
   5 workload type (0 training, 1 inference)    6 log-scaled parameter count    7 isolated throughput T_j(c)
   8 micro-batch size   9 activation checkpointing flag   10 mixed-precision flag
  11 ISL               12 OSL                              13 prefix caching ratio
A training job's inference slots and an inference job's training slots hold 0.

Pair (i, j), predicting the slowdown of i next to j: x[0:14] = f_i, x[14:28] = f_j, then the 8 pairwise
features (Sec. 3.3.1):
  28-31 the mean over the two jobs of SM Active, SM Occupancy, DRAM Active, Tensor Core Active
  32    co-location type: type_i + type_j (0 training-training, 1 training-inference, 2 inference-inference)
  33    memory pressure (fb_i + fb_j) / C_mem
  34    compute balance min(sm_i, sm_j) / max(sm_i, sm_j), 1 when both are 0
  35    memory intensity difference |dram_i / sm_i - dram_j / sm_j|, a term with sm = 0 counting as 0
Readings: the paper counts 8 pairwise features but names 5 hardware metrics whose means enter; the
means are taken over the four utilization metrics (fractions of cycles), the framebuffer entering
through the memory pressure ratio, which gives the stated 36. A zero SM Active (undefined ratios)
takes the values above.

Network (Sec. 3.3.2, inference mode: dropout is the identity, Batch Normalization uses its running
statistics):  h1 = ReLU(BN1(W1 x + b1)),  h2 = ReLU(BN2(W2 h1 + b2)),  S_hat = 1 + ReLU(W3 h2 + b3)
(Eq. dnn_pred), BN(z) = gamma (z - mean) / sqrt(var + eps) + beta per unit. Parameters are given in
fp32 (as a trained model stores them) and used exactly, converted to fp64.
"""

from __future__ import annotations

import dataclasses

import numpy as np

N_JOB = 14
N_PAIR = 8
N_FEAT = 2 * N_JOB + N_PAIR

SM_ACTIVE, SM_OCC, DRAM_ACTIVE, FB_USED, TC_ACTIVE, WTYPE = 0, 1, 2, 3, 4, 5
UTILIZATION = (SM_ACTIVE, SM_OCC, DRAM_ACTIVE, TC_ACTIVE)


@dataclasses.dataclass
class IacModel:
    """Parameters of the network: W1 (H, 36), b1 (H), bn1 (4, H) = gamma, beta, running mean,
    running variance; W2 (H, H), b2 (H), bn2 (4, H); W3 (H), b3 scalar; eps of both BN layers."""

    W1: np.ndarray
    b1: np.ndarray
    bn1: np.ndarray
    W2: np.ndarray
    b2: np.ndarray
    bn2: np.ndarray
    W3: np.ndarray
    b3: float
    eps: float

    @property
    def H(self) -> int:
        return int(self.W1.shape[0])


def pair_features(f_i: np.ndarray, f_j: np.ndarray, c_mem: float) -> np.ndarray:
    """The 36 features of the pair (i, j) (Sec. 3.3.1), fp64."""
    a = np.asarray(f_i, dtype=np.float64)
    b = np.asarray(f_j, dtype=np.float64)
    x = np.zeros(N_FEAT)
    x[0:N_JOB] = a
    x[N_JOB:2 * N_JOB] = b
    k = 2 * N_JOB
    for m in UTILIZATION:                       # aggregate contention per utilization metric
        x[k] = (a[m] + b[m]) / 2.0
        k += 1
    x[k] = a[WTYPE] + b[WTYPE]                  # co-location type
    x[k + 1] = (a[FB_USED] + b[FB_USED]) / float(c_mem)   # proximity to the memory ceiling
    sm_lo, sm_hi = min(a[SM_ACTIVE], b[SM_ACTIVE]), max(a[SM_ACTIVE], b[SM_ACTIVE])
    x[k + 2] = 1.0 if sm_hi == 0.0 else sm_lo / sm_hi      # symmetry of SM demand

    def intensity(f):
        return 0.0 if f[SM_ACTIVE] == 0.0 else f[DRAM_ACTIVE] / f[SM_ACTIVE]

    x[k + 3] = abs(intensity(a) - intensity(b))             # compute- vs memory-bound complementarity
    return x


def feature_matrix(job_features: np.ndarray, pairs: np.ndarray, c_mem: float) -> np.ndarray:
    """Rows pair_features(job_features[i], job_features[j]) for every pair (i, j)."""
    jf = np.asarray(job_features, dtype=np.float64).reshape(-1, N_JOB)
    pr = np.asarray(pairs, dtype=np.int64).reshape(-1, 2)
    out = np.empty((pr.shape[0], N_FEAT))
    for p, (i, j) in enumerate(pr):
        out[p] = pair_features(jf[i], jf[j], c_mem)
    return out


def batch_norm(z: np.ndarray, bn: np.ndarray, eps: float) -> np.ndarray:
    """Batch Normalization at inference (running statistics), per unit (last axis)."""
    gamma, beta, mean, var = (np.asarray(bn[q], dtype=np.float64) for q in range(4))
    return gamma * (z - mean) / np.sqrt(var + float(eps)) + beta


def relu(z: np.ndarray) -> np.ndarray:
    return np.maximum(z, 0.0)


def forward(x: np.ndarray, m: IacModel) -> np.ndarray:
    """S_hat of Eq. dnn_pred for feature rows x (n, 36)."""
    x = np.asarray(x, dtype=np.float64)
    f64 = lambda a: np.asarray(a, dtype=np.float64)
    h1 = relu(batch_norm(x @ f64(m.W1).T + f64(m.b1), m.bn1, m.eps))
    h2 = relu(batch_norm(h1 @ f64(m.W2).T + f64(m.b2), m.bn2, m.eps))
    return 1.0 + relu(h2 @ f64(m.W3) + float(m.b3))


def predict(job_features: np.ndarray, pairs: np.ndarray, c_mem: float, m: IacModel) -> np.ndarray:
    """Predicted slowdown S_hat_{i|j} of every pair (i, j)."""
    return forward(feature_matrix(job_features, pairs, c_mem), m)
