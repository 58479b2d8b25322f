"""The oracle over every scenario of a benchmark workload, in a pool of processes.

Each worker regenerates its own scenario (the generator's draws are counter based, so scenario s alone
is bit-identical to scenario s of the full batch) and runs the oracle's tatonnement on it with every
trace. The pool is started with the `spawn` method, so it is safe to create after the parent process
has used the GPU. Results are cached on disk (ESP_ORACLE_CACHE, default ~/.cache/esp_oracle) under a
key that covers the oracle's and the generator's sources, the workload, the scenario and the solve
parameters; a cache that cannot be written is skipped. The cache only saves time: a missing or
unreadable entry is recomputed.
"""

from __future__ import annotations

import hashlib
import os
import sys

import numpy as np

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

FIELDS = ("lam", "sel", "demand", "min_score", "lambda_trace", "demand_trace", "selhash_trace", "dual_trace")
SCALARS = ("rounds_run", "converged", "feasible", "status", "primal", "dual", "best_dual")


def _sources_digest() -> str:
    h = hashlib.sha256()
    for rel in ("oracle/esp_oracle.c", "oracle/esp_oracle.h", "oracle/__init__.py",
                "paper_2608_07971_gb300/workloads.py"):
        with open(os.path.join(ROOT, rel), "rb") as f:
            h.update(f.read())
    return h.hexdigest()


def _cache_dir():
    d = os.environ.get("ESP_ORACLE_CACHE") or os.path.join(os.path.expanduser("~"), ".cache", "esp_oracle")
    try:
        os.makedirs(d, exist_ok=True)
        return d
    except OSError:
        return None


def solve_one(job):
    """Worker: (workload name, scenario, rounds, sources digest) -> dict of the oracle's solution."""
    name, s, T, digest = job
    if ROOT not in sys.path:
        sys.path.insert(0, ROOT)
    d = _cache_dir()
    path = None
    if d is not None:
        key = hashlib.sha256(f"{digest}|{name}|{s}|{T}".encode()).hexdigest()[:32]
        path = os.path.join(d, f"{name}_{s}_{T}_{key}.npz")
        try:
            with np.load(path) as z:
                return {k: z[k] for k in z.files}
        except Exception:
            pass
    import oracle
    from paper_2608_07971_gb300 import workloads as W
    w = W.make(name, scenarios=[s])
    ref = oracle.solve_scenario(w.table, 0, w.eta0, T, mode=w.mode, step=w.step, traces=True)
    out = {k: np.asarray(getattr(ref, k)) for k in FIELDS}
    out.update({k: np.asarray(getattr(ref, k)) for k in SCALARS})
    if path is not None:
        try:
            tmp = path + f".{os.getpid()}.tmp.npz"
            np.savez(tmp, **out)
            os.replace(tmp, path)
        except Exception:
            pass
    return out


class Batch:
    """Starts the oracle on the given scenarios in the background; result() waits for all of them."""

    def __init__(self, name: str, scenarios, rounds: int, workers=None):
        import concurrent.futures as cf
        import multiprocessing as mp
        self.scenarios = list(scenarios)
        digest = _sources_digest()
        import oracle
        oracle.build()     # once, here: the workers only load it
        n = workers or max(1, min(len(self.scenarios), os.cpu_count() or 1))
        self.ex = cf.ProcessPoolExecutor(max_workers=n, mp_context=mp.get_context("spawn"))
        self.futs = [self.ex.submit(solve_one, (name, s, rounds, digest)) for s in self.scenarios]

    def result(self):
        try:
            return {s: f.result() for s, f in zip(self.scenarios, self.futs)}
        finally:
            self.ex.shutdown()
