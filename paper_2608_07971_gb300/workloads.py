"""Seeded synthetic option tables for the ESP tatonnement (Sec. 3.1's profiles p = (R_j(c), T_j(c), L_j)).

This module only draws inputs: it holds none of the solver's arithmetic. Both the CUDA path and the
oracle consume the arrays it returns.

Random numbers are counter based. Draw ``n`` of stream ``(seed, stream)`` is SplitMix64's output
number ``n`` for the start state ``mix(seed * GAMMA ^ stream)`` (Steele, Lea and Flood, "Fast
splittable pseudorandom number generators", OOPSLA 2014), so every draw is computed directly from
(seed, scenario, job, configuration, field). A subset of scenarios is therefore bit-identical to the
same scenarios of the full batch, which lets tests check a full-size batch scenario by scenario.

Workloads (the paper's own traces and profiles are not available; these stand in for its
training/inference job mix, Sec. 5.1, with the shapes the benchmark configurations name):
  tiny_cluster        S=1,    J=64,    K=8,   R=4           eta 0.05, T=200,  seed 1
  cluster_512         S=1,    J=2048,  K=16,  R=6           eta 0.02, T=500,  seed 2
  whatif_batch        S=1024, J=2048,  K=16,  R=6 (jitter)  eta 0.02, T=300,  seed 3
  placement_expanded  S=1,    J=4096,  K=768 (12 x 64 nodes), R=8, P=134      T=400, seed 4
  heavy_tail          S=16,   J=65536, K=min(256, Zipf 1.3), R=6             T=1000, seed 5
"""

from __future__ import annotations

import dataclasses
from typing import Optional, Sequence

import numpy as np

GAMMA = np.uint64(0x9E3779B97F4A7C15)
_M1 = np.uint64(0xBF58476D1CE4E5B9)
_M2 = np.uint64(0x94D049BB133111EB)

# Stream tags, so per-job, per-node, matrix and capacity draws never share a stream.
_TAG_NODE = np.uint64(1 << 62)
_TAG_MATRIX = np.uint64(1 << 61)
_TAG_CAP = np.uint64(1 << 60)
_TAG_IAC = np.uint64(1 << 59)

# Field numbers inside a job's stream; configuration k uses 16 + 8k + field.
F_BASE_Z1, F_BASE_Z2, F_MEM, F_CPU, F_HOST, F_NVL, F_NET, F_K, F_TYPE, F_SENS = range(10)
C_GPU, C_CKPT, C_MEMSCALE, C_MULT = range(4)

RAW, NORMALIZED = 0, 1
STEP_FIXED, STEP_INV_SQRT = 0, 1


def _mix(z: np.ndarray) -> np.ndarray:
    z = (z ^ (z >> np.uint64(30))) * _M1
    z = (z ^ (z >> np.uint64(27))) * _M2
    return z ^ (z >> np.uint64(31))


def draw_bits(seed: int, stream: np.ndarray, counter) -> np.ndarray:
    """64 random bits: SplitMix64 output number ``counter`` of stream ``stream``."""
    stream = np.asarray(stream, dtype=np.uint64)
    with np.errstate(over="ignore"):
        state = _mix((np.uint64(seed) * GAMMA) ^ stream)
        ctr = np.asarray(counter, dtype=np.uint64) + np.uint64(1)
        return _mix(state + ctr * GAMMA)


def uniform(seed, stream, counter) -> np.ndarray:
    """Uniform double in [0, 1) with 53 random bits."""
    return (draw_bits(seed, stream, counter) >> np.uint64(11)).astype(np.float64) * 2.0**-53


def randint(seed, stream, counter, lo: int, hi: int) -> np.ndarray:
    """Uniform integer in [lo, hi] from the top 32 bits (multiply-shift, no division)."""
    n = np.uint64(hi - lo + 1)
    top = draw_bits(seed, stream, counter) >> np.uint64(32)
    return (np.int64(lo) + ((top * n) >> np.uint64(32)).astype(np.int64))


def normal(seed, stream, c1, c2) -> np.ndarray:
    """Standard normal by Box-Muller from two uniforms."""
    u1 = uniform(seed, stream, c1)
    u2 = uniform(seed, stream, c2)
    return np.sqrt(-2.0 * np.log1p(-u1)) * np.cos(2.0 * np.pi * u2)


@dataclasses.dataclass
class OptionTable:
    """S independent scenarios of J jobs; options of a job are contiguous (job-major CSR).

    units[o, r] is R_j(c)[r] (int32 >= 0), values[o] is w_j T_j(c) (fp64, larger is better),
    job_off[s*J + j] .. job_off[s*J + j + 1] are job (s, j)'s global option indices, capacity[s, k]
    is C_k of scenario s. With group given, stored columns r >= r_global of option o are priced by
    lambda[r_global + (R - r_global) * group[o] + (r - r_global)].
    """

    S: int
    J: int
    R: int
    P: int
    r_global: int
    job_off: np.ndarray
    units: np.ndarray
    values: np.ndarray
    group: Optional[np.ndarray]
    capacity: np.ndarray

    @property
    def n_opt(self) -> int:
        return int(self.job_off[-1])

    def option_counts(self) -> np.ndarray:
        return np.diff(self.job_off)

    def table_bytes(self) -> int:
        """Bytes of the option table a full evaluation pass must read (units + values [+ group])."""
        per = 4 * self.R + 8 + (2 if self.group is not None else 0)
        return self.n_opt * per

    def digest(self) -> str:
        """SHA-256 of the table: shape, then job offsets, units, values, group column and capacities
        as little-endian bytes, so that two runs (or two arms of a benchmark) can show they read the
        same synthetic table."""
        import hashlib
        h = hashlib.sha256()
        h.update(np.asarray([self.S, self.J, self.R, self.P, self.r_global, self.group is not None], "<i8").tobytes())
        for a, dt in ((self.job_off, "<i8"), (self.units, "<i4"), (self.values, "<f8"), (self.capacity, "<i8")):
            h.update(np.ascontiguousarray(a, dt).tobytes())
        if self.group is not None:
            h.update(np.ascontiguousarray(self.group, "<u2").tobytes())
        return h.hexdigest()

    def scenario(self, s: int) -> "OptionTable":
        """Scenario s alone, re-based to option index 0."""
        a, b = int(self.job_off[s * self.J]), int(self.job_off[(s + 1) * self.J])
        return OptionTable(
            S=1, J=self.J, R=self.R, P=self.P, r_global=self.r_global,
            job_off=self.job_off[s * self.J:(s + 1) * self.J + 1] - a,
            units=self.units[a:b], values=self.values[a:b],
            group=None if self.group is None else self.group[a:b],
            capacity=self.capacity[s:s + 1].copy())


@dataclasses.dataclass
class Workload:
    name: str
    table: OptionTable
    eta0: float
    rounds: int
    step: int = STEP_FIXED
    mode: int = NORMALIZED
    seed: int = 0
    factors: Optional["PlacementFactors"] = None   # placement_expanded: the table before expansion


@dataclasses.dataclass
class PlacementFactors:
    """A placement-expanded table in factored form: option (k, n) of job j (local index k * N + n)
    has the units of configuration k (columns r >= r_global priced per node n) and the value
    cfg_values[j, k] - (double)(sens[j] *fp32 D[job_type[j], node_type[n]])."""
    S: int
    J: int
    KC: int                   # configurations per job
    N: int                    # nodes
    R: int
    r_global: int
    cfg_units: np.ndarray     # (S*J, KC, R) int32
    cfg_values: np.ndarray    # (S*J, KC) fp64
    sens: np.ndarray          # (S*J,) fp32
    job_type: np.ndarray      # (S*J,) int32
    node_type: np.ndarray     # (N,) int32
    D: np.ndarray             # (NT, NT) fp32
    capacity: np.ndarray      # (S, r_global + (R - r_global) * N) int64


# Capacities (Sec. 5.1's testbed scaled to the named clusters): GPU milli-share, GPU memory MiB,
# CPU millicores, host memory MiB, NVLink units, network units.
CAP_TINY = [64000, 64 * 81920, 512000, 64 * 1048576]
CAP_512 = [8 * c for c in CAP_TINY] + [512 * 900, 512 * 400]
NODES = 64
CAP_NODE = [8000, 8 * 81920]


def _job_profile(seed, stream, R):
    """Per-job draws: base value b_j (log-normal), memory, CPU, host memory, NVLink, network."""
    b = np.exp(normal(seed, stream, F_BASE_Z1, F_BASE_Z2))
    mem = randint(seed, stream, F_MEM, 1024, 163840)
    cpu = randint(seed, stream, F_CPU, 1000, 64000)
    host = randint(seed, stream, F_HOST, 4096, 524288)
    nvl = randint(seed, stream, F_NVL, 0, 900)
    net = randint(seed, stream, F_NET, 0, 400)
    return b, mem, cpu, host, nvl, net


def _configs(seed, job_stream, k, b, mem, cpu, host, nvl, net, R, out_units=None, out_values=None):
    """Configuration k of each job (vectorised over options): GPU share 1000*U{1..8}; half are
    checkpointing-like (memory x U[0.4, 1], value x U[0.7, 1]); value b_j * sqrt(g / 8000) * mult.
    Columns: GPU share, GPU memory, CPU, host memory [, NVLink, network] (the last four scale with
    the GPU share, host memory does not)."""
    n = len(k)
    units = np.empty((n, R), dtype=np.int32) if out_units is None else out_units
    c = np.uint64(16) + np.uint64(8) * k.astype(np.uint64)
    g = 1000 * randint(seed, job_stream, c + np.uint64(C_GPU), 1, 8)
    ck = (draw_bits(seed, job_stream, c + np.uint64(C_CKPT)) >> np.uint64(63)).astype(bool)
    scale = 0.4 + 0.6 * uniform(seed, job_stream, c + np.uint64(C_MEMSCALE))
    mult = 0.7 + 0.3 * uniform(seed, job_stream, c + np.uint64(C_MULT))
    frac = g.astype(np.float64) / 8000.0
    units[:, 0] = g
    units[:, 1] = np.where(ck, np.maximum(1, np.rint(mem * scale)), mem)
    units[:, 2] = np.maximum(1000, np.rint(cpu * frac))
    units[:, 3] = host
    if R >= 6:
        units[:, 4] = np.rint(nvl * frac)
        units[:, 5] = np.rint(net * frac)
    value = b * np.sqrt(frac) * np.where(ck, mult, 1.0)
    if out_values is not None:
        out_values[:] = value
        value = out_values
    return units, value


def _zipf_counts(seed, stream, s_exp=1.3, kmax=256):
    """K_j = min(kmax, X), P(X = k) proportional to k^-s_exp for k >= 1 (the clipped reading)."""
    n = 100000
    k = np.arange(1, n, dtype=np.float64)
    zeta = np.sum(k ** -s_exp) + n ** (1 - s_exp) / (s_exp - 1) + 0.5 * n ** -s_exp \
        + s_exp * n ** (-s_exp - 1) / 12
    cdf = np.cumsum(np.arange(1, kmax, dtype=np.float64) ** -s_exp / zeta)
    u = uniform(seed, stream, F_K)
    return np.minimum(kmax, np.searchsorted(cdf, u, side="right") + 1).astype(np.int64)


def _lower_median_per_job(col: np.ndarray, job_of_opt: np.ndarray, job_off_local: np.ndarray):
    """Lower median (element (K-1)//2 in sorted order) of col within each job."""
    key = (job_of_opt.astype(np.int64) << np.int64(32)) | col.astype(np.int64)
    key.sort()
    K = np.diff(job_off_local)
    pick = key[job_off_local[:-1] + (K - 1) // 2]
    return pick & np.int64(0xFFFFFFFF)


_BLOCK = 1 << 15


def _build(seed, scenarios, J, R, K_of_job):
    """Common option construction, one scenario at a time (bounded temporaries).
    Returns job_off (int64), units (int32, n_opt x R), values (fp64)."""
    scen = np.asarray(scenarios, dtype=np.int64)
    S = len(scen)
    js = np.arange(J, dtype=np.uint64)
    streams = [(np.uint64(s) << np.uint64(32)) | js for s in scen]
    Ks = [K_of_job(st) for st in streams]
    job_off = np.zeros(S * J + 1, dtype=np.int64)
    np.cumsum(np.concatenate(Ks) if S else np.zeros(0, np.int64), out=job_off[1:])
    n_opt = int(job_off[-1])
    units = np.empty((n_opt, R), dtype=np.int32)
    values = np.empty(n_opt, dtype=np.float64)

    def one(si):
        K, st = Ks[si], streams[si]
        a, b = int(job_off[si * J]), int(job_off[(si + 1) * J])
        loc = job_off[si * J:(si + 1) * J + 1] - a
        job_idx = np.repeat(np.arange(J, dtype=np.int64), K)
        bj, mem, cpu, host, nvl, net = _job_profile(seed, st, R)
        for c0 in range(0, b - a, _BLOCK):  # cache-sized blocks of options
            c1 = min(b - a, c0 + _BLOCK)
            ji = job_idx[c0:c1]
            k_local = np.arange(c0, c1, dtype=np.int64) - loc[:-1][ji]
            _configs(seed, st[ji], k_local, bj[ji], mem[ji], cpu[ji], host[ji], nvl[ji], net[ji], R,
                     units[a + c0:a + c1], values[a + c0:a + c1])

    # scenarios write disjoint slices; numpy releases the GIL inside its array loops, so threads
    # overlap them (every draw is a function of its counter: the result does not depend on the order)
    if S > 1 and n_opt > (1 << 20):
        from concurrent.futures import ThreadPoolExecutor
        import os
        with ThreadPoolExecutor(max_workers=min(S, os.cpu_count() or 1, 16)) as ex:
            list(ex.map(one, range(S)))
    else:
        for si in range(S):
            one(si)
    return job_off, units, values


def tiny_cluster(scenarios: Optional[Sequence[int]] = None) -> Workload:
    seed, J, R = 1, 64, 4
    scenarios = [0] if scenarios is None else scenarios
    job_off, units, value = _build(seed, scenarios, J, R, lambda st: np.full(st.shape, 8, np.int64))
    S = len(scenarios)
    cap = np.tile(np.asarray(CAP_TINY, dtype=np.int64), (S, 1))
    t = OptionTable(S, J, R, R, R, job_off, units, value, None, cap)
    return Workload("tiny_cluster", t, eta0=0.05, rounds=200, seed=seed)


def cluster_512(scenarios: Optional[Sequence[int]] = None, J: int = 2048) -> Workload:
    seed, R = 2, 6
    scenarios = [0] if scenarios is None else scenarios
    job_off, units, value = _build(seed, scenarios, J, R, lambda st: np.full(st.shape, 16, np.int64))
    S = len(scenarios)
    cap = np.tile(np.asarray(CAP_512, dtype=np.int64), (S, 1))
    t = OptionTable(S, J, R, R, R, job_off, units, value, None, cap)
    return Workload("cluster_512", t, eta0=0.02, rounds=500, seed=seed)


def whatif_batch(scenarios: Optional[Sequence[int]] = None, J: int = 2048) -> Workload:
    """1024 independent cluster_512-shaped scenarios; capacity of (s, r) jittered by U[0.8, 1.2]."""
    seed, R = 3, 6
    scenarios = list(range(1024)) if scenarios is None else list(scenarios)
    job_off, units, value = _build(seed, scenarios, J, R, lambda st: np.full(st.shape, 16, np.int64))
    S = len(scenarios)
    cap_stream = _TAG_CAP | np.asarray(scenarios, dtype=np.uint64)
    jit = 0.8 + 0.4 * uniform(seed, cap_stream[:, None], np.arange(R, dtype=np.uint64)[None, :])
    cap = np.rint(np.asarray(CAP_512, dtype=np.float64)[None, :] * jit).astype(np.int64)
    t = OptionTable(S, J, R, R, R, job_off, units, value, None, cap)
    return Workload("whatif_batch", t, eta0=0.02, rounds=300, seed=seed)


def placement_expanded(scenarios: Optional[Sequence[int]] = None, J: int = 4096) -> Workload:
    """Options = 12 configurations x 64 node slots (local index k*64 + n). Columns 6-7 repeat the GPU
    share and GPU memory of configuration k, priced per node n (group = n). The value of (k, n) is
    v_k minus the fp32 interference penalty sigma_j * D[a_j][b_n] (Sec. 3.3's slowdown folded into
    the value), with D a symmetric 64x64 Beta(2, 8) matrix (2nd order statistic of 9 uniforms)."""
    seed, R, KC = 4, 8, 12
    scenarios = [0] if scenarios is None else list(scenarios)
    scen = np.asarray(scenarios, dtype=np.int64)
    S = len(scen)
    js = np.arange(J, dtype=np.int64)
    job_stream = ((scen[:, None].astype(np.uint64) << np.uint64(32)) | js[None, :].astype(np.uint64)).ravel()
    nj = S * J
    b, mem, cpu, host, nvl, net = _job_profile(seed, job_stream, 6)
    kk = np.tile(np.arange(KC, dtype=np.int64), nj)
    jj = np.repeat(np.arange(nj, dtype=np.int64), KC)
    cols12, v12 = _configs(seed, job_stream[jj], kk, b[jj], mem[jj], cpu[jj], host[jj], nvl[jj], net[jj], 6)
    cols12 = cols12.astype(np.int32)
    cols12 = cols12.reshape(nj, KC, 6)
    v12 = v12.reshape(nj, KC)

    # Pairwise degradation matrix and node / job types.
    a_idx, b_idx = np.triu_indices(NODES)
    mstream = _TAG_MATRIX | (a_idx.astype(np.uint64) * np.uint64(NODES) + b_idx.astype(np.uint64))
    u9 = np.stack([uniform(seed, mstream, c) for c in range(9)], axis=1)
    d_upper = np.sort(u9, axis=1)[:, 1].astype(np.float32)
    D = np.zeros((NODES, NODES), dtype=np.float32)
    D[a_idx, b_idx] = d_upper
    D[b_idx, a_idx] = d_upper
    node_type = randint(seed, _TAG_NODE | np.arange(NODES, dtype=np.uint64), 0, 0, NODES - 1)
    job_type = randint(seed, job_stream, F_TYPE, 0, NODES - 1)
    sens = uniform(seed, job_stream, F_SENS).astype(np.float32)
    penalty = (sens[:, None] * D[job_type][:, node_type]).astype(np.float32)  # fp32 product

    units = np.empty((nj, KC, NODES, R), dtype=np.int32)
    units[:, :, :, :6] = cols12[:, :, None, :]
    units[:, :, :, 6] = cols12[:, :, None, 0]
    units[:, :, :, 7] = cols12[:, :, None, 1]
    values = v12[:, :, None] - penalty[:, None, :].astype(np.float64)
    group = np.broadcast_to(np.arange(NODES, dtype=np.uint16)[None, None, :], (nj, KC, NODES))
    job_off = np.arange(nj + 1, dtype=np.int64) * (KC * NODES)
    P = 6 + 2 * NODES
    cap_row = np.asarray(CAP_512 + CAP_NODE * NODES, dtype=np.int64)
    cap = np.tile(cap_row, (S, 1))
    t = OptionTable(S, J, R, P, 6, job_off, units.reshape(-1, R), values.reshape(-1),
                    np.ascontiguousarray(group.reshape(-1)), cap)
    cfg_units = np.empty((nj, KC, R), dtype=np.int32)
    cfg_units[:, :, :6] = cols12
    cfg_units[:, :, 6] = cols12[:, :, 0]
    cfg_units[:, :, 7] = cols12[:, :, 1]
    factors = PlacementFactors(S, J, KC, NODES, R, 6, cfg_units, np.ascontiguousarray(v12, np.float64), sens,
                               job_type.astype(np.int32), node_type.astype(np.int32), D, cap)
    return Workload("placement_expanded", t, eta0=0.02, rounds=400, seed=seed, factors=factors)


def heavy_tail(scenarios: Optional[Sequence[int]] = None, J: int = 65536) -> Workload:
    """K_j = min(256, Zipf(1.3)); capacity C_r = floor(0.6 * sum_j lower-median_c u_{j,c,r}) per scenario,
    so the cluster is oversubscribed."""
    seed, R = 5, 6
    scenarios = list(range(16)) if scenarios is None else list(scenarios)
    job_off, units, value = _build(seed, scenarios, J, R, lambda st: _zipf_counts(seed, st))
    S = len(scenarios)
    cap = np.zeros((S, R), dtype=np.int64)

    def one(si):
        a, b = int(job_off[si * J]), int(job_off[(si + 1) * J])
        loc_off = job_off[si * J:(si + 1) * J + 1] - a
        loc_job = np.repeat(np.arange(J, dtype=np.int64), np.diff(loc_off))
        for r in range(R):
            med = _lower_median_per_job(units[a:b, r], loc_job, loc_off)
            cap[si, r] = (6 * int(med.sum())) // 10

    # scenarios are independent (numpy's sort releases the GIL, so threads overlap them)
    from concurrent.futures import ThreadPoolExecutor
    import os
    with ThreadPoolExecutor(max_workers=max(1, min(S, os.cpu_count() or 1, 16))) as ex:
        list(ex.map(one, range(S)))
    cap = np.maximum(cap, 1)
    t = OptionTable(S, J, R, R, R, job_off, units, value, None, cap)
    return Workload("heavy_tail", t, eta0=0.02, rounds=1000, seed=seed)


# ---- IAC co-location pairs (Sec. 3.3.1) ---------------------------------------------------------
#
# Profile rows of 14 features per (job, configuration), row index j*K + k, in the order of
# Sec. 3.3.1: SM Active, SM Occupancy, DRAM Active, Framebuffer Used (MB), Tensor Core Active,
# workload type (0 training, 1 inference), log-scaled parameter count, isolated throughput,
# micro-batch, checkpointing flag, mixed-precision flag, ISL, OSL, prefix caching ratio. The
# paper's profiled co-location experiments are not available; these draws give each feature a
# plausible range (type, parameter count and the task-level attributes are per job, the hardware
# metrics and throughput per configuration).

IAC_ROW = 14
IAC_C_MEM = 81920.0     # MB: an 80 GB device, the paper's example capacity
# Approximate mean and standard deviation of each of the 36 network inputs under these draws (the
# pairwise block from two independent rows); used only to scale the synthetic weights.
IAC_INPUT_MEAN = np.asarray([0.55, 0.36, 0.475, 40024, 0.45, 0.5, 22, 1.13, 5.25, 0.25, 0.4, 2080, 516, 0.225] * 2 +
                            [0.55, 0.36, 0.475, 0.45, 1.0, 0.977, 0.6, 1.5])
IAC_INPUT_STD = np.asarray([0.26, 0.2, 0.245, 21925, 0.26, 0.5, 2.31, 0.6, 8.0, 0.43, 0.49, 2700, 660, 0.3] * 2 +
                           [0.18, 0.14, 0.17, 0.18, 0.71, 0.38, 0.25, 2.0])


def iac_rows(seed: int, J: int, K: int) -> np.ndarray:
    """(J*K, 14) fp32 profile rows."""
    js = np.repeat(np.arange(J, dtype=np.uint64), K)
    ks = np.tile(np.arange(K, dtype=np.uint64), J)
    job = _TAG_IAC | js
    cfg = _TAG_IAC | (np.uint64(1) << np.uint64(40)) | (js * np.uint64(K) + ks)
    f = np.zeros((J * K, IAC_ROW), np.float64)
    wtype = randint(seed, job, 0, 0, 1)
    f[:, 0] = 0.1 + 0.9 * uniform(seed, cfg, 0)
    f[:, 1] = f[:, 0] * (0.3 + 0.7 * uniform(seed, cfg, 1))
    f[:, 2] = 0.05 + 0.85 * uniform(seed, cfg, 2)
    f[:, 3] = randint(seed, cfg, 3, 2048, 78000)
    f[:, 4] = 0.9 * uniform(seed, cfg, 4)
    f[:, 5] = wtype
    f[:, 6] = 18.0 + 8.0 * uniform(seed, job, 1)
    f[:, 7] = np.exp(0.5 * normal(seed, cfg, 5, 6))
    train = wtype == 0
    f[:, 8] = np.where(train, 2.0 ** randint(seed, job, 2, 0, 5), 0.0)
    f[:, 9] = np.where(train, randint(seed, cfg, 7, 0, 1), 0)
    f[:, 10] = np.where(train, (uniform(seed, job, 3) < 0.8).astype(np.float64), 0.0)
    f[:, 11] = np.where(train, 0, randint(seed, job, 4, 128, 8192))
    f[:, 12] = np.where(train, 0, randint(seed, job, 5, 16, 2048))
    f[:, 13] = np.where(train, 0.0, 0.9 * uniform(seed, cfg, 8))
    return f.astype(np.float32)


def iac_pairs(seed: int, S: int, J: int, K: int) -> np.ndarray:
    """(S*J*K, 2) int32: for what-if scenario s, every configuration k of every job j (row j*K + k)
    against its co-located partner's current configuration: partner (j + 1 + d) mod J with
    d ~ U{0..J-2}, at configuration c ~ U{0..K-1}, drawn per (s, j)."""
    s = np.repeat(np.arange(S, dtype=np.uint64), J)
    j = np.tile(np.arange(J, dtype=np.uint64), S)
    st = _TAG_IAC | (np.uint64(2) << np.uint64(40)) | (s << np.uint64(20)) | j
    d = randint(seed, st, 0, 0, max(J - 2, 0))
    c = randint(seed, st, 1, 0, K - 1)
    partner = ((j.astype(np.int64) + 1 + d) % J) * K + c
    out = np.empty((S * J, K, 2), np.int32)
    out[:, :, 0] = (j.astype(np.int64) * K)[:, None] + np.arange(K)[None, :]
    out[:, :, 1] = partner[:, None]
    return out.reshape(-1, 2)


@dataclasses.dataclass
class IacParams:
    """Synthetic parameters of the IAC network (the trained weights are not available): W1 (H, 36),
    b1 (H), bn1 (4, H) = gamma, beta, running mean, running variance; W2 (H, H), b2, bn2; W3 (H), b3;
    eps. W1 is scaled per input by the inputs' spread so that the first layer sees inputs of order
    one, as a trained first layer would."""

    W1: np.ndarray
    b1: np.ndarray
    bn1: np.ndarray
    W2: np.ndarray
    b2: np.ndarray
    bn2: np.ndarray
    W3: np.ndarray
    b3: float
    eps: float


def iac_model(seed: int, H: int = 64, eps: float = 1e-5) -> IacParams:
    def nrm(layer, n):
        st = _TAG_IAC | (np.uint64(3 + layer) << np.uint64(40)) | np.arange(n, dtype=np.uint64)
        return normal(seed, st, 0, 1)

    def uni(layer, n, lo, hi):
        st = _TAG_IAC | (np.uint64(3 + layer) << np.uint64(40)) | np.arange(n, dtype=np.uint64)
        return lo + (hi - lo) * uniform(seed, st, 2)

    n_in = 2 * IAC_ROW + 8
    W1 = nrm(0, H * n_in).reshape(H, n_in) * np.sqrt(2.0 / n_in) / IAC_INPUT_STD
    b1 = -(W1 @ IAC_INPUT_MEAN) + 0.1 * nrm(1, H)          # inputs centred on their mean
    bn1 = np.stack([uni(2, H, 0.8, 1.2), 0.2 * nrm(3, H), 0.1 * nrm(4, H), uni(5, H, 0.8, 1.5)])
    W2 = nrm(6, H * H).reshape(H, H) * np.sqrt(2.0 / H)
    b2 = 0.1 * nrm(7, H)
    bn2 = np.stack([uni(8, H, 0.8, 1.2), 0.2 * nrm(9, H), 0.3 * nrm(10, H), uni(11, H, 0.8, 1.5)])
    W3 = np.abs(nrm(12, H)) * np.sqrt(2.0 / H) * np.where(np.arange(H) % 2 == 0, 1.0, -1.0)
    f32 = lambda a: np.ascontiguousarray(a, np.float32)
    return IacParams(W1=f32(W1), b1=f32(b1), bn1=f32(bn1), W2=f32(W2), b2=f32(b2), bn2=f32(bn2), W3=f32(W3),
                     b3=float(np.float32(0.05)), eps=eps)


@dataclasses.dataclass
class IacWorkload:
    name: str
    rows: np.ndarray
    pairs: np.ndarray
    c_mem: float
    model: IacParams
    S: int
    J: int
    K: int


def iac_batch(S: int = 1024, J: int = 2048, K: int = 16, H: int = 64, seed: int = 6) -> IacWorkload:
    """IAC slowdowns for S what-if scenarios of the 512-GPU cluster's shape (J=2048 jobs, K=16
    configurations): every option against its partner, S*J*K pairs (33.5 M at the defaults)."""
    return IacWorkload("iac_whatif", iac_rows(seed, J, K), iac_pairs(seed, S, J, K), IAC_C_MEM,
                       iac_model(seed, H), S, J, K)


WORKLOADS = {
    "tiny_cluster": tiny_cluster,
    "cluster_512": cluster_512,
    "whatif_batch": whatif_batch,
    "placement_expanded": placement_expanded,
    "heavy_tail": heavy_tail,
}


def make(name: str, **kw) -> Workload:
    return WORKLOADS[name](**kw)


def random_table(rng: np.random.Generator, S: int, J: int, R: int, kmin: int, kmax: int,
                 umax: int = 100, cap_frac: float = 0.5, dyadic: bool = False,
                 groups: int = 0, r_global: Optional[int] = None) -> OptionTable:
    """Small random table for tests: K_j ~ U{kmin..kmax}, units U{0..umax}, values log-normal or, with
    dyadic=True, multiples of 1/8 so that every sum and product of the method is exact in fp64."""
    K = rng.integers(kmin, kmax + 1, size=S * J)
    job_off = np.zeros(S * J + 1, dtype=np.int64)
    np.cumsum(K, out=job_off[1:])
    n = int(job_off[-1])
    units = rng.integers(0, umax + 1, size=(n, R)).astype(np.int32)
    if dyadic:
        values = rng.integers(0, 64, size=n).astype(np.float64) / 8.0
    else:
        values = np.exp(rng.standard_normal(n))
    group = None
    if groups:
        rg = R - 1 if r_global is None else r_global
        P = rg + (R - rg) * groups
        group = rng.integers(0, groups, size=n).astype(np.uint16)
    else:
        rg, P = R, R
    # Capacity: cap_frac of J mean-sized demands; a per-group column is shared by fewer jobs.
    per_col = np.full(P, cap_frac * J * umax / 2.0)
    if groups:
        per_col[rg:] /= groups
    cap = np.tile(np.maximum(1, per_col.astype(np.int64)), (S, 1))
    return OptionTable(S, J, R, P, rg, job_off, units, values, group, cap)
