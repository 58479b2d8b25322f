"""Runs the oracle's pins and a set of seeded solves against a given build of the oracle library and
saves every output array (test infrastructure; tests/test_host_sanitized.py runs it in a child
process with a build instrumented by AddressSanitizer and UndefinedBehaviorSanitizer, and runs
run_cases in-process with the plain build to compare).

    python -m tests.sanitized_oracle_run LIB OUT.npz [--pins]
"""

from __future__ import annotations

import sys

import numpy as np

import oracle
from paper_2608_07971_gb300 import workloads as W


def cases():
    """(name, table, eta0, rounds, mode, step, tol, with lambda0): the workload shapes (uniform,
    heavy-tailed, grouped placement, small cluster) at reduced sizes, and ragged random tables with
    1-option jobs, a tolerance and a warm start."""
    rng = np.random.default_rng(31)
    out = []
    w = W.tiny_cluster()
    out.append(("tiny", w.table, w.eta0, 40, w.mode, w.step, 0.0, False))
    w = W.whatif_batch(scenarios=[0, 5], J=192)
    out.append(("whatif", w.table, w.eta0, 25, w.mode, w.step, 0.0, False))
    w = W.heavy_tail(scenarios=[1], J=1024)
    out.append(("heavy", w.table, w.eta0, 12, w.mode, w.step, 0.0, False))
    w = W.placement_expanded(scenarios=[0], J=48)
    out.append(("placement", w.table, w.eta0, 10, w.mode, w.step, 0.0, False))
    w = W.cluster_512(scenarios=[3], J=256)
    out.append(("cluster", w.table, w.eta0, 20, w.mode, oracle.STEP_INV_SQRT, 0.0, False))
    out.append(("ragged_raw", W.random_table(rng, 3, 57, 5, 1, 40), 0.002, 30, oracle.RAW,
                oracle.STEP_INV_SQRT, 0.0, True))
    out.append(("ragged_tol", W.random_table(rng, 2, 33, 3, 1, 9, groups=4), 0.05, 200, oracle.NORMALIZED,
                oracle.STEP_FIXED, 1e-3, True))
    out.append(("ones", W.random_table(rng, 2, 20, 2, 1, 1), 0.1, 5, oracle.NORMALIZED, oracle.STEP_FIXED,
                0.0, False))
    return out


def run_cases(lib) -> dict:
    """Every oracle entry point on every case; returns name -> array."""
    rng = np.random.default_rng(32)
    res = {}
    for name, t, eta0, T, mode, step, tol, warm in cases():
        ot = oracle.OracleTable(t)
        for s in range(t.S):
            l0 = rng.random(t.P) * 0.5 if warm else None
            r = oracle.solve_scenario(ot, s, eta0, T, mode, step, tol, l0, traces=True, sel_trace=True, lib=lib)
            key = f"{name}/{s}"
            for f in ("lam", "sel", "demand", "min_score", "lambda_trace", "demand_trace", "selhash_trace",
                      "dual_trace", "sel_trace"):
                res[f"{key}/{f}"] = np.asarray(getattr(r, f))
            res[f"{key}/scalars"] = np.array([r.rounds_run, r.converged, r.feasible, r.status, r.primal,
                                              r.dual, r.best_dual])
            lam = rng.random(t.P)
            sel, dem, ms = oracle.best_response(ot, s, lam, mode, lib=lib)
            p = oracle.effective_prices(ot, s, lam, mode, lib=lib)
            o = int(t.job_off[s * t.J])
            res[f"{key}/br"] = np.concatenate([sel, dem, ms, p,
                                               [oracle.reduced_cost(ot, o, p, lib=lib),
                                                oracle.dual_value(ot, s, lam, ms, mode, lib=lib),
                                                oracle.selection_hash(sel, lib=lib) & 0xFFFFFFFF]])
            lam2, st = oracle.price_update(ot, s, 3, dem, lam, eta0, mode, step, lib=lib)
            res[f"{key}/update"] = np.concatenate([lam2, [st]])
        n = t.n_opt
        c_cur = rng.integers(-1, 3, t.S * t.J).astype(np.int32)
        s_hat = 1.0 + rng.random(n)
        tau = 1.0 + 0.5 * rng.random(t.S * t.J)
        res[f"{name}/penalized"] = oracle.penalized_values(ot, 0.03, c_cur, 0.7, s_hat, tau, lib=lib)
        res[f"{name}/penalty"] = np.array([oracle.penalty(c, cc, 0.03, 0.7, sh, ta, lib=lib)
                                           for c, cc, sh, ta in ((0, 1, 1.4, 1.2), (2, 2, 1.1, 1.2), (1, -1, 2.0, 1.5))])
    K = rng.integers(1, 6, 30)
    q_off = np.zeros(31, np.int64)
    q_off[1:] = np.cumsum(K)
    q_units = rng.integers(0, 500, (int(q_off[-1]), 4)).astype(np.int32)
    cap = rng.integers(2000, 9000, 4).astype(np.int64)
    res["capacity"] = np.concatenate([oracle.effective_capacity(cap, q_off, q_units, g, lib=lib)
                                      for g in (0.0, 0.5, 1.0, 3.0)])
    res["threshold"] = np.array([oracle.adaptive_threshold(1.1, 0.3, u, 0.8, 0.1, lib=lib)
                                 for u in (0.2, 0.8, 0.95, 2.0)])
    return res


def main(argv) -> int:
    lib_path, out = argv[1], argv[2]
    lib = oracle.load(lib_path)
    if "--pins" in argv:
        from tests import test_oracle_mutants as mut
        failures = mut.failing_pins(lib)
        if failures:
            print(f"{failures} pins failed", file=sys.stderr)
            return 1
    np.savez(out, **run_cases(lib))
    return 0


if __name__ == "__main__":
    sys.exit(main(sys.argv))
