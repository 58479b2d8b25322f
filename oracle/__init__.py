"""ctypes wrapper around the C oracle (esp_oracle.c) of the ESP tatonnement, Sec. 3.2.

TEST INFRASTRUCTURE: only tests/, __graft_entry__.smoke() and bench.py's CPU-baseline and reference
legs may import this package. It imports nothing from the library under paper_2608_07971_gb300/; it
reads any table object with the fields of workloads.OptionTable.
"""

from __future__ import annotations

import ctypes
import dataclasses
import os
import subprocess
from typing import Optional, Sequence

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "esp_oracle.c")
_LIB = os.path.join(_HERE, "liboracle.so")
CFLAGS = ["-O2", "-ffp-contract=off", "-std=c11", "-fPIC", "-shared", "-Wall"]

RAW, NORMALIZED = 0, 1
STEP_FIXED, STEP_INV_SQRT = 0, 1


def build(force: bool = False, extra_flags: Sequence[str] = (), out: Optional[str] = None) -> str:
    """Compile esp_oracle.c with gcc; returns the shared library path."""
    out = out or _LIB
    if force or not os.path.exists(out) or os.path.getmtime(out) < max(
            os.path.getmtime(_SRC), os.path.getmtime(os.path.join(_HERE, "esp_oracle.h"))):
        cc = os.environ.get("CC", "gcc")
        subprocess.check_call([cc, *CFLAGS, *extra_flags, _SRC, "-o", out, "-lm"])
    return out


class _Table(ctypes.Structure):
    _fields_ = [("S", ctypes.c_int32), ("J", ctypes.c_int32), ("R", ctypes.c_int32),
                ("P", ctypes.c_int32), ("r_global", ctypes.c_int32),
                ("job_off", ctypes.c_void_p), ("units", ctypes.c_void_p),
                ("values", ctypes.c_void_p), ("group", ctypes.c_void_p),
                ("capacity", ctypes.c_void_p)]


class _Params(ctypes.Structure):
    _fields_ = [("eta0", ctypes.c_double), ("step", ctypes.c_int32), ("mode", ctypes.c_int32),
                ("max_rounds", ctypes.c_int32), ("tol", ctypes.c_double)]


class _Result(ctypes.Structure):
    _fields_ = [("rounds_run", ctypes.c_int32), ("converged", ctypes.c_int32),
                ("feasible", ctypes.c_int32), ("status", ctypes.c_int32),
                ("primal", ctypes.c_double), ("dual", ctypes.c_double),
                ("best_dual", ctypes.c_double)]


_lib_cache = {}


def load(path: Optional[str] = None):
    path = path or build()
    if path in _lib_cache:
        return _lib_cache[path]
    lib = ctypes.CDLL(path)
    vp, i32, i64, dbl = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64, ctypes.c_double
    T = ctypes.POINTER(_Table)
    lib.esp_oracle_price_index.argtypes = [T, i64, i32]
    lib.esp_oracle_price_index.restype = i32
    lib.esp_oracle_effective_prices.argtypes = [T, i32, i32, vp, vp]
    lib.esp_oracle_reduced_cost.argtypes = [T, i64, vp]
    lib.esp_oracle_reduced_cost.restype = dbl
    lib.esp_oracle_best_response.argtypes = [T, i32, i32, vp, vp, vp, vp]
    lib.esp_oracle_dual_value.argtypes = [T, i32, i32, vp, vp]
    lib.esp_oracle_dual_value.restype = dbl
    lib.esp_oracle_price_update.argtypes = [T, i32, ctypes.POINTER(_Params), i32, vp, vp, vp]
    lib.esp_oracle_price_update.restype = ctypes.c_int
    lib.esp_oracle_selection_hash.argtypes = [i32, vp]
    lib.esp_oracle_selection_hash.restype = ctypes.c_uint64
    lib.esp_oracle_solve.argtypes = [T, i32, ctypes.POINTER(_Params), vp, vp, vp, vp, vp,
                                     ctypes.POINTER(_Result), vp, vp, vp, vp, vp]
    lib.esp_oracle_solve.restype = ctypes.c_int
    lib.esp_oracle_adaptive_threshold.argtypes = [dbl, dbl, dbl, dbl, dbl]
    lib.esp_oracle_adaptive_threshold.restype = dbl
    lib.esp_oracle_penalty.argtypes = [i32, i32, dbl, dbl, dbl, dbl]
    lib.esp_oracle_penalty.restype = dbl
    lib.esp_oracle_penalized_values.argtypes = [T, dbl, vp, dbl, vp, vp, vp]
    lib.esp_oracle_effective_capacity.argtypes = [i32, vp, i32, vp, vp, dbl, vp]
    _lib_cache[path] = lib
    return lib


def _ptr(a: Optional[np.ndarray]):
    return None if a is None else a.ctypes.data


class OracleTable:
    """Keeps contiguous copies of an OptionTable's arrays alive behind the C struct."""

    def __init__(self, table):
        self.table = table
        self.job_off = np.ascontiguousarray(table.job_off, dtype=np.int64)
        self.units = np.ascontiguousarray(table.units, dtype=np.int32)
        self.values = np.ascontiguousarray(table.values, dtype=np.float64)
        self.group = None if table.group is None else np.ascontiguousarray(table.group, dtype=np.uint16)
        self.capacity = np.ascontiguousarray(table.capacity, dtype=np.int64)
        self.c = _Table(table.S, table.J, table.R, table.P, table.r_global, _ptr(self.job_off),
                        _ptr(self.units), _ptr(self.values), _ptr(self.group), _ptr(self.capacity))


@dataclasses.dataclass
class ScenarioSolution:
    lam: np.ndarray
    sel: np.ndarray
    demand: np.ndarray
    min_score: np.ndarray
    rounds_run: int
    converged: int
    feasible: int
    status: int
    primal: float
    dual: float
    best_dual: float
    lambda_trace: Optional[np.ndarray] = None
    demand_trace: Optional[np.ndarray] = None
    selhash_trace: Optional[np.ndarray] = None
    dual_trace: Optional[np.ndarray] = None
    sel_trace: Optional[np.ndarray] = None


def solve_scenario(table, s: int, eta0: float, rounds: int, mode: int = NORMALIZED,
                   step: int = STEP_FIXED, tol: float = 0.0,
                   lambda0: Optional[np.ndarray] = None, traces: bool = False,
                   sel_trace: bool = False, lib=None) -> ScenarioSolution:
    """Run the tatonnement of scenario s (esp_oracle_solve)."""
    lib = lib or load()
    ot = table if isinstance(table, OracleTable) else OracleTable(table)
    t = ot.table
    P, J, T = t.P, t.J, rounds
    prm = _Params(eta0, step, mode, T, tol)
    lam = np.zeros(P); sel = np.zeros(J, np.int32); dem = np.zeros(P, np.int64)
    ms = np.zeros(J)
    l0 = None if lambda0 is None else np.ascontiguousarray(lambda0, dtype=np.float64)
    lt = np.full((T + 1, P), np.nan) if traces else None
    dt = np.zeros((T, P), np.int64) if traces else None
    ht = np.zeros(T, np.uint64) if traces else None
    gt = np.full(T + 1, np.nan) if traces else None
    st = np.zeros((T, J), np.int32) if sel_trace else None
    res = _Result()
    lib.esp_oracle_solve(ctypes.byref(ot.c), s, ctypes.byref(prm), _ptr(l0), _ptr(lam), _ptr(sel),
                         _ptr(dem), _ptr(ms), ctypes.byref(res), _ptr(lt), _ptr(dt), _ptr(ht),
                         _ptr(gt), _ptr(st))
    return ScenarioSolution(lam, sel, dem, ms, res.rounds_run, res.converged, res.feasible,
                            res.status, res.primal, res.dual, res.best_dual, lt, dt, ht, gt, st)


def best_response(table, s: int, lam: np.ndarray, mode: int = NORMALIZED, lib=None):
    """Selection, demand and minimal reduced costs of scenario s at prices lam."""
    lib = lib or load()
    ot = table if isinstance(table, OracleTable) else OracleTable(table)
    t = ot.table
    sel = np.zeros(t.J, np.int32); dem = np.zeros(t.P, np.int64); ms = np.zeros(t.J)
    lam = np.ascontiguousarray(lam, dtype=np.float64)
    lib.esp_oracle_best_response(ctypes.byref(ot.c), s, mode, _ptr(lam), _ptr(sel), _ptr(dem), _ptr(ms))
    return sel, dem, ms


def reduced_cost(table, o: int, p: np.ndarray, lib=None) -> float:
    lib = lib or load()
    ot = table if isinstance(table, OracleTable) else OracleTable(table)
    p = np.ascontiguousarray(p, dtype=np.float64)
    return lib.esp_oracle_reduced_cost(ctypes.byref(ot.c), o, _ptr(p))


def effective_prices(table, s: int, lam: np.ndarray, mode: int, lib=None) -> np.ndarray:
    lib = lib or load()
    ot = table if isinstance(table, OracleTable) else OracleTable(table)
    lam = np.ascontiguousarray(lam, dtype=np.float64)
    p = np.zeros(ot.table.P)
    lib.esp_oracle_effective_prices(ctypes.byref(ot.c), s, mode, _ptr(lam), _ptr(p))
    return p


def dual_value(table, s: int, lam: np.ndarray, min_score: np.ndarray, mode: int, lib=None) -> float:
    lib = lib or load()
    ot = table if isinstance(table, OracleTable) else OracleTable(table)
    lam = np.ascontiguousarray(lam, dtype=np.float64)
    ms = np.ascontiguousarray(min_score, dtype=np.float64)
    return lib.esp_oracle_dual_value(ctypes.byref(ot.c), s, mode, _ptr(lam), _ptr(ms))


def price_update(table, s: int, t1: int, demand: np.ndarray, lam: np.ndarray, eta0: float,
                 mode: int = NORMALIZED, step: int = STEP_FIXED, lib=None):
    lib = lib or load()
    ot = table if isinstance(table, OracleTable) else OracleTable(table)
    prm = _Params(eta0, step, mode, 0, 0.0)
    dem = np.ascontiguousarray(demand, dtype=np.int64)
    lam = np.ascontiguousarray(lam, dtype=np.float64)
    out = np.zeros(ot.table.P)
    st = lib.esp_oracle_price_update(ctypes.byref(ot.c), s, ctypes.byref(prm), t1, _ptr(dem), _ptr(lam), _ptr(out))
    return out, st


def selection_hash(sel: np.ndarray, lib=None) -> int:
    lib = lib or load()
    sel = np.ascontiguousarray(sel, dtype=np.int32)
    return int(lib.esp_oracle_selection_hash(len(sel), _ptr(sel)))


def solve(table, eta0: float, rounds: int, mode: int = NORMALIZED, step: int = STEP_FIXED,
          tol: float = 0.0, lambda0: Optional[np.ndarray] = None, traces: bool = False,
          scenarios: Optional[Sequence[int]] = None):
    """Solve every (or the listed) scenario one after the other on this thread."""
    ot = OracleTable(table)
    lib = load()
    out = []
    for s in (range(table.S) if scenarios is None else scenarios):
        l0 = None if lambda0 is None else lambda0[s]
        out.append(solve_scenario(ot, s, eta0, rounds, mode, step, tol, l0, traces, lib=lib))
    return out


def adaptive_threshold(tau_base: float, beta: float, util: float, util_target: float, beta_max: float,
                       lib=None) -> float:
    """tau_j(t) of Eq. adaptive_threshold."""
    return (lib or load()).esp_oracle_adaptive_threshold(tau_base, beta, util, util_target, beta_max)


def penalty(c: int, c_cur: int, gamma0: float, alpha: float, s_hat: float, tau: float, lib=None) -> float:
    """Gamma_j(c) of Eq. esp_score: switching cost plus interference penalty."""
    return (lib or load()).esp_oracle_penalty(c, c_cur, gamma0, alpha, s_hat, tau)


def penalized_values(table, gamma0: float = 0.0, c_cur=None, alpha: float = 0.0, s_hat=None, tau=None,
                     lib=None) -> np.ndarray:
    """v - Gamma for every option (Eq. esp_score with the Gamma term)."""
    lib = lib or load()
    ot = table if isinstance(table, OracleTable) else OracleTable(table)
    out = np.zeros(ot.values.size)
    cc = None if c_cur is None else np.ascontiguousarray(c_cur, np.int32)
    sh = None if s_hat is None else np.ascontiguousarray(s_hat, np.float64)
    ta = None if tau is None else np.ascontiguousarray(tau, np.float64)
    lib.esp_oracle_penalized_values(ctypes.byref(ot.c), gamma0, _ptr(cc), alpha, _ptr(sh), _ptr(ta), _ptr(out))
    return out


def effective_capacity(capacity, q_off, q_units, gamma: float, lib=None) -> np.ndarray:
    """C_eff of Eq. effective_capacity (componentwise minimum footprint of each queued job)."""
    lib = lib or load()
    cap = np.ascontiguousarray(capacity, np.int64)
    qo = np.ascontiguousarray(q_off, np.int64)
    qu = np.ascontiguousarray(q_units, np.int32)
    R = cap.size
    out = np.zeros(R, np.int64)
    lib.esp_oracle_effective_capacity(R, _ptr(cap), qo.size - 1, _ptr(qo), _ptr(qu), gamma, _ptr(out))
    return out

