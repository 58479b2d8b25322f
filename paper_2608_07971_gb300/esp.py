"""Thin ctypes binding of libesp.so (include/esp.h). Argument marshalling only: every step of the
solve runs in the library's CUDA kernels. The binding fails loudly when the library is missing.

Functions keep the C names (esp_create, esp_load_options, esp_solve, ...). ``Solver`` bundles them
for numpy / torch callers.
"""

from __future__ import annotations

import ctypes
import dataclasses
import os
from typing import Optional

import numpy as np

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "libesp.so")

ESP_OK, ESP_ERR_INVALID_ARG, ESP_ERR_OVERFLOW, ESP_ERR_OOM, ESP_ERR_CUDA = 0, 1, 2, 3, 4
ESP_ERR_NOT_LOADED, ESP_ERR_TIMEOUT, ESP_ERR_STATE, ESP_ERR_UNSUPPORTED = 5, 6, 7, 8
ESP_PRICE_RAW, ESP_PRICE_NORMALIZED = 0, 1
ESP_STEP_FIXED, ESP_STEP_INV_SQRT = 0, 1
ESP_FLAG_EXACT_ONLY, ESP_FLAG_PER_ROUND_LAUNCH, ESP_FLAG_PASS_EVENTS, ESP_FLAG_RESIDENT = 0x1, 0x2, 0x4, 0x8

EXPORTED = [
    "esp_create", "esp_set_stream", "esp_load_options", "esp_load_options_device", "esp_solve",
    "esp_solve_async", "esp_get_result", "esp_get_prices", "esp_get_selection", "esp_get_demand",
    "esp_evaluate", "esp_last_launch_count", "esp_pass_times", "esp_status_string", "esp_destroy",
    "esp_debug_tile_options", "esp_debug_plan", "esp_debug_stats", "esp_debug_resident",
    "esp_debug_sort_layout", "esp_debug_plan_runs", "esp_debug_set_sorted_layout", "esp_debug_set_pdl", "esp_debug_set_plan_waves",
    "esp_debug_hold_barrier", "esp_debug_set_wait_limit", "esp_debug_hold_stage", "esp_debug_fail_alloc",
    "esp_debug_pass_kernel", "esp_debug_set_interleave", "esp_debug_set_stage_f32",
    "esp_debug_set_persistent", "esp_debug_persistent", "esp_debug_persist_waits",
    "esp_debug_load_profile",
    "esp_evaluate_noalloc",
    "esp_set_penalties", "esp_adaptive_threshold", "esp_effective_capacity", "esp_load_placement",
    "esp_iac_create", "esp_iac_set_stream", "esp_iac_load_model", "esp_iac_predict", "esp_iac_predict_host",
    "esp_iac_last_launch_count", "esp_iac_destroy", "esp_iac_set_path", "esp_iac_synchronize",
    "esp_iac_debug_set_wait_limit", "esp_iac_debug_hold_commit",
]


class EspError(RuntimeError):
    def __init__(self, status: int, what: str):
        self.status = status
        super().__init__(f"{what}: {esp_status_string(status)} ({status})")


class esp_params(ctypes.Structure):
    _fields_ = [("eta0", ctypes.c_double), ("step", ctypes.c_int32), ("mode", ctypes.c_int32),
                ("max_rounds", ctypes.c_int32), ("flags", ctypes.c_uint32), ("tol", ctypes.c_double),
                ("lambda0", ctypes.c_void_p), ("lambda_trace", ctypes.c_void_p),
                ("demand_trace", ctypes.c_void_p), ("selhash_trace", ctypes.c_void_p),
                ("dual_trace", ctypes.c_void_p), ("round_time_trace", ctypes.c_void_p)]


class esp_result(ctypes.Structure):
    _fields_ = [("rounds_run", ctypes.c_int32), ("converged", ctypes.c_int32),
                ("feasible", ctypes.c_int32), ("status", ctypes.c_int32),
                ("primal", ctypes.c_double), ("dual", ctypes.c_double), ("best_dual", ctypes.c_double),
                ("device_ms", ctypes.c_float)]


_lib = None


def load_library(path: Optional[str] = None):
    """Loads libesp.so (build it with paper_2608_07971_gb300.build.build()). Raises if missing."""
    global _lib
    if _lib is not None and path is None:
        return _lib
    path = path or LIB_PATH
    if not os.path.exists(path):
        raise RuntimeError(f"libesp.so not found at {path}; run paper_2608_07971_gb300.build.build() "
                           "(there is no CPU fallback)")
    lib = ctypes.CDLL(path)
    vp, i32, u32, i64 = ctypes.c_void_p, ctypes.c_int32, ctypes.c_uint32, ctypes.c_int64
    st = ctypes.c_int
    sig = {
        "esp_create": ([ctypes.POINTER(vp), ctypes.c_int, vp], st),
        "esp_set_stream": ([vp, vp], st),
        "esp_load_options": ([vp, i32, i32, i32, i32, i32, vp, vp, vp, vp, vp], st),
        "esp_load_options_device": ([vp, i32, i32, i32, i32, i32, vp, vp, vp, vp, vp], st),
        "esp_solve": ([vp, ctypes.POINTER(esp_params), vp], st),
        "esp_solve_async": ([vp, ctypes.POINTER(esp_params)], st),
        "esp_get_result": ([vp, vp], st),
        "esp_get_prices": ([vp, vp], st),
        "esp_get_selection": ([vp, vp], st),
        "esp_get_demand": ([vp, vp], st),
        "esp_evaluate": ([vp, vp, i32, u32, vp, vp, vp], st),
        "esp_last_launch_count": ([vp, ctypes.POINTER(i64)], st),
        "esp_pass_times": ([vp, ctypes.POINTER(ctypes.c_double), ctypes.POINTER(i64), i32], st),
        "esp_status_string": ([st], ctypes.c_char_p),
        "esp_destroy": ([vp], None),
        "esp_debug_tile_options": ([i32, i32], i32),
        "esp_debug_stats": ([vp, ctypes.POINTER(i64), ctypes.POINTER(i64), i32], st),
        "esp_debug_resident": ([vp, i32, ctypes.POINTER(i32), ctypes.POINTER(i32)], st),
        "esp_debug_sort_layout": ([vp, i32, i32, vp, vp, vp, vp], st),
        "esp_debug_plan_runs": ([vp, vp, vp, i32, i32, i32, i32, vp, i32, vp, i32, ctypes.POINTER(i32),
                                 ctypes.POINTER(i32)], st),
        "esp_debug_set_sorted_layout": ([vp, i32], st),
        "esp_debug_set_pdl": ([vp, i32], st),
        "esp_debug_set_plan_waves": ([vp, i32], st),
        "esp_debug_hold_barrier": ([vp], st),
        "esp_debug_set_wait_limit": ([vp, u32], st),
        "esp_debug_hold_stage": ([vp], st),
        "esp_debug_fail_alloc": ([vp, i64], st),
        "esp_debug_pass_kernel": ([vp, ctypes.POINTER(i32)], st),
        "esp_debug_set_interleave": ([vp, i32], st),
        "esp_debug_set_stage_f32": ([vp, i32], st),
        "esp_debug_set_persistent": ([vp, i32], st),
        "esp_debug_persistent": ([vp, ctypes.POINTER(i32)], st),
        "esp_debug_persist_waits": ([vp, ctypes.POINTER(i64), ctypes.POINTER(i64), i32], st),
        "esp_debug_load_profile": ([vp, ctypes.POINTER(ctypes.c_double), ctypes.POINTER(i64), ctypes.POINTER(i64)],
                                   st),
        "esp_set_penalties": ([vp, ctypes.c_double, vp, ctypes.c_double, vp, vp], st),
        "esp_load_placement": ([vp, i32, i32, i32, i32, i32, i32, vp, vp, vp, vp, i32, vp, vp, vp], st),
        "esp_adaptive_threshold": ([i64, vp, ctypes.c_double, ctypes.c_double, ctypes.c_double, ctypes.c_double, vp],
                                   st),
        "esp_effective_capacity": ([i32, vp, i32, vp, vp, ctypes.c_double, vp], st),
        "esp_debug_plan": ([vp, i32, i32, i32, i32, vp, i32, vp, i32, ctypes.POINTER(i32), ctypes.POINTER(i32)], st),
        "esp_evaluate_noalloc": ([i32, i32, i32, vp, vp, vp, vp, vp, i32, vp, vp, vp, vp], st),
        "esp_iac_create": ([ctypes.POINTER(vp), ctypes.c_int, vp], st),
        "esp_iac_set_stream": ([vp, vp], st),
        "esp_iac_load_model": ([vp, i32, vp, vp, vp, vp, vp, vp, vp, ctypes.c_float, ctypes.c_float], st),
        "esp_iac_predict": ([vp, i32, vp, i64, vp, ctypes.c_float, vp], st),
        "esp_iac_predict_host": ([vp, i32, vp, i64, vp, ctypes.c_float, vp], st),
        "esp_iac_last_launch_count": ([vp, ctypes.POINTER(i64)], st),
        "esp_iac_destroy": ([vp], None),
        "esp_iac_set_path": ([vp, i32], st),
        "esp_iac_synchronize": ([vp], st),
        "esp_iac_debug_set_wait_limit": ([vp, u32], st),
        "esp_iac_debug_hold_commit": ([vp], st),
    }
    for name, (args, res) in sig.items():
        fn = getattr(lib, name)
        fn.argtypes = args
        fn.restype = res
    if path == LIB_PATH or _lib is None:
        _lib = lib
    return lib


def esp_status_string(status: int) -> str:
    return load_library().esp_status_string(status).decode()


def _check(status: int, what: str, ok=(ESP_OK,)):
    if status not in ok:
        raise EspError(status, what)
    return status


def _p(a) -> Optional[int]:
    """Address of a numpy array or torch tensor (None for None)."""
    if a is None:
        return None
    if isinstance(a, np.ndarray):
        return a.ctypes.data
    return int(a.data_ptr())


# --- the C calls, same names -------------------------------------------------------------------

def esp_create(device: int = -1, stream: Optional[int] = None) -> int:
    h = ctypes.c_void_p()
    _check(load_library().esp_create(ctypes.byref(h), device, stream), "esp_create")
    return h.value


def esp_set_stream(ctx: int, stream: Optional[int]) -> None:
    _check(load_library().esp_set_stream(ctx, stream), "esp_set_stream")


def esp_load_options(ctx, S, J, R, P, r_global, job_offsets, units, values, group, capacity) -> None:
    _check(load_library().esp_load_options(ctx, S, J, R, P, r_global, _p(job_offsets), _p(units), _p(values),
                                           _p(group), _p(capacity)), "esp_load_options")


def esp_load_options_device(ctx, S, J, R, P, r_global, job_offsets, units, values, group, capacity) -> None:
    _check(load_library().esp_load_options_device(ctx, S, J, R, P, r_global, _p(job_offsets), _p(units),
                                                  _p(values), _p(group), _p(capacity)),
           "esp_load_options_device")


def esp_solve(ctx: int, params: esp_params, results) -> int:
    return _check(load_library().esp_solve(ctx, ctypes.byref(params), _p(results)), "esp_solve",
                  ok=(ESP_OK, ESP_ERR_OVERFLOW))


def esp_solve_async(ctx: int, params: esp_params) -> None:
    _check(load_library().esp_solve_async(ctx, ctypes.byref(params)), "esp_solve_async")


def esp_get_result(ctx: int, results) -> int:
    return _check(load_library().esp_get_result(ctx, _p(results)), "esp_get_result", ok=(ESP_OK, ESP_ERR_OVERFLOW))


def esp_get_prices(ctx: int, out) -> None:
    _check(load_library().esp_get_prices(ctx, _p(out)), "esp_get_prices")


def esp_get_selection(ctx: int, out) -> None:
    _check(load_library().esp_get_selection(ctx, _p(out)), "esp_get_selection")


def esp_get_demand(ctx: int, out) -> None:
    _check(load_library().esp_get_demand(ctx, _p(out)), "esp_get_demand")


def esp_evaluate(ctx: int, lam, mode: int, flags: int, sel, demand, min_score) -> None:
    _check(load_library().esp_evaluate(ctx, _p(lam), mode, flags, _p(sel), _p(demand), _p(min_score)),
           "esp_evaluate")


def esp_last_launch_count(ctx: int) -> int:
    n = ctypes.c_int64()
    _check(load_library().esp_last_launch_count(ctx, ctypes.byref(n)), "esp_last_launch_count")
    return n.value


def esp_pass_times(ctx: int, reset: bool = True):
    """(summed milliseconds, number) of the evaluation passes timed with ESP_FLAG_PASS_EVENTS."""
    ms, n = ctypes.c_double(), ctypes.c_int64()
    _check(load_library().esp_pass_times(ctx, ctypes.byref(ms), ctypes.byref(n), 1 if reset else 0),
           "esp_pass_times")
    return ms.value, n.value


def esp_evaluate_noalloc(S, J, R, job_offsets, units, values, capacity, lam, mode, sel, demand, min_score,
                         stream: Optional[int] = None) -> None:
    """Best response that allocates nothing (device tensors in and out; see include/esp.h)."""
    _check(load_library().esp_evaluate_noalloc(S, J, R, _p(job_offsets), _p(units), _p(values), _p(capacity),
                                               _p(lam), mode, _p(sel), _p(demand), _p(min_score), stream),
           "esp_evaluate_noalloc")


def esp_debug_stats(ctx: int, reset: bool = True):
    """(exact resolutions since the last reset, duplicates marked at load)."""
    r, m = ctypes.c_int64(), ctypes.c_int64()
    _check(load_library().esp_debug_stats(ctx, ctypes.byref(r), ctypes.byref(m), 1 if reset else 0),
           "esp_debug_stats")
    return r.value, m.value


def esp_debug_resident(ctx: int, force_cs: int = 0):
    """(cluster size, co-resident clusters) of the resident kernel for the loaded table; force_cs
    1/2/4/8/16 forces that size for later solves, 0 restores the automatic choice. None when the
    table cannot run resident."""
    cs, nc = ctypes.c_int32(), ctypes.c_int32()
    status = load_library().esp_debug_resident(ctx, int(force_cs), ctypes.byref(cs), ctypes.byref(nc))
    if status == ESP_ERR_UNSUPPORTED:
        return None
    _check(status, "esp_debug_resident")
    return cs.value, nc.value


def esp_load_placement(ctx: int, f) -> None:
    """Loads a workloads.PlacementFactors-like factored placement table (see include/esp.h)."""
    arrs = [np.ascontiguousarray(f.cfg_units, np.int32), np.ascontiguousarray(f.cfg_values, np.float64),
            np.ascontiguousarray(f.sens, np.float32), np.ascontiguousarray(f.job_type, np.int32),
            np.ascontiguousarray(f.node_type, np.int32), np.ascontiguousarray(f.D, np.float32),
            np.ascontiguousarray(f.capacity, np.int64)]
    NT = int(arrs[5].shape[0])
    _check(load_library().esp_load_placement(ctx, f.S, f.J, f.KC, f.N, f.R, f.r_global, _p(arrs[0]), _p(arrs[1]),
                                             _p(arrs[2]), _p(arrs[3]), NT, _p(arrs[4]), _p(arrs[5]), _p(arrs[6])),
           "esp_load_placement")


def esp_set_penalties(ctx: int, gamma0: float = 0.0, c_cur=None, alpha: float = 0.0, s_hat=None, tau=None) -> None:
    """Gamma term of Eq. esp_score for later solves (see include/esp.h)."""
    cc = None if c_cur is None else np.ascontiguousarray(c_cur, np.int32)
    sh = None if s_hat is None else np.ascontiguousarray(s_hat, np.float64)
    ta = None if tau is None else np.ascontiguousarray(tau, np.float64)
    _check(load_library().esp_set_penalties(ctx, float(gamma0), _p(cc), float(alpha), _p(sh), _p(ta)),
           "esp_set_penalties")


def esp_adaptive_threshold(tau_base, beta: float, util: float, util_target: float, beta_max: float) -> np.ndarray:
    """tau_j(t) of Eq. adaptive_threshold (host)."""
    tb = np.ascontiguousarray(tau_base, np.float64)
    out = np.zeros_like(tb)
    _check(load_library().esp_adaptive_threshold(tb.size, _p(tb), beta, util, util_target, beta_max, _p(out)),
           "esp_adaptive_threshold")
    return out


def esp_effective_capacity(capacity, q_offsets, q_units, gamma: float) -> np.ndarray:
    """C_eff of Eq. effective_capacity (host)."""
    cap = np.ascontiguousarray(capacity, np.int64)
    qo = np.ascontiguousarray(q_offsets, np.int64)
    qu = np.ascontiguousarray(q_units, np.int32)
    out = np.zeros(cap.size, np.int64)
    _check(load_library().esp_effective_capacity(cap.size, _p(cap), qo.size - 1, _p(qo), _p(qu), gamma, _p(out)),
           "esp_effective_capacity")
    return out


def esp_destroy(ctx: int) -> None:
    load_library().esp_destroy(ctx)


# --- convenience ---------------------------------------------------------------------------------

RESULT_DTYPE = np.dtype([("rounds_run", np.int32), ("converged", np.int32), ("feasible", np.int32),
                         ("status", np.int32), ("primal", np.float64), ("dual", np.float64),
                         ("best_dual", np.float64), ("device_ms", np.float32)], align=True)
assert RESULT_DTYPE.itemsize == ctypes.sizeof(esp_result)


@dataclasses.dataclass
class Solution:
    lam: np.ndarray          # S x P
    sel: np.ndarray          # S x J
    demand: np.ndarray       # S x P
    result: np.ndarray       # S records of RESULT_DTYPE
    status: int
    lambda_trace: Optional[np.ndarray] = None   # S x (T+1) x P
    demand_trace: Optional[np.ndarray] = None   # S x T x P
    selhash_trace: Optional[np.ndarray] = None  # S x T
    dual_trace: Optional[np.ndarray] = None     # S x (T+1)
    round_time_trace: Optional[np.ndarray] = None  # S x T, GPU global timer (ns) of each round's update


class Solver:
    """A context holding one option table (workloads.OptionTable-like) on the GPU."""

    def __init__(self, table=None, device: int = -1, stream: Optional[int] = None):
        self.ctx = esp_create(device, stream)
        self.shape = None
        if table is not None:
            self.load(table)

    def close(self):
        if self.ctx:
            esp_destroy(self.ctx)
            self.ctx = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def load(self, t):
        arrs = dict(job_off=np.ascontiguousarray(t.job_off, np.int64),
                    units=np.ascontiguousarray(t.units, np.int32),
                    values=np.ascontiguousarray(t.values, np.float64),
                    group=None if t.group is None else np.ascontiguousarray(t.group, np.uint16),
                    cap=np.ascontiguousarray(t.capacity, np.int64))
        esp_load_options(self.ctx, t.S, t.J, t.R, t.P, t.r_global, arrs["job_off"], arrs["units"],
                         arrs["values"], arrs["group"], arrs["cap"])
        self.shape = (t.S, t.J, t.R, t.P)

    def load_placement(self, f):
        """Factored placement table (workloads.PlacementFactors)."""
        esp_load_placement(self.ctx, f)
        self.shape = (f.S, f.J, f.R, f.r_global + (f.R - f.r_global) * f.N)

    def load_device(self, S, J, R, P, r_global, job_off, units, values, group, cap):
        """Table given as device tensors (torch); copied device-to-device."""
        esp_load_options_device(self.ctx, S, J, R, P, r_global, job_off, units, values, group, cap)
        self.shape = (S, J, R, P)

    def params(self, eta0, rounds, mode=ESP_PRICE_NORMALIZED, step=ESP_STEP_FIXED, tol=0.0, flags=0,
               lambda0=None) -> esp_params:
        prm = esp_params()
        prm.eta0, prm.step, prm.mode, prm.max_rounds, prm.flags, prm.tol = eta0, step, mode, rounds, flags, tol
        prm.lambda0 = _p(lambda0)
        return prm

    def solve(self, eta0, rounds, mode=ESP_PRICE_NORMALIZED, step=ESP_STEP_FIXED, tol=0.0, flags=0,
              lambda0=None, traces=False) -> Solution:
        S, J, R, P = self.shape
        T = rounds
        l0 = None if lambda0 is None else np.ascontiguousarray(lambda0, np.float64).reshape(S, P)
        prm = self.params(eta0, rounds, mode, step, tol, flags, l0)
        lt = dt = ht = gt = tt = None
        if traces:          # True: every trace; "prices": the price, demand and round-time trajectories
            lt = np.full((S, T + 1, P), np.nan)
            dt = np.zeros((S, T, P), np.int64)
            tt = np.zeros((S, T), np.uint64)
            prm.lambda_trace, prm.demand_trace, prm.round_time_trace = _p(lt), _p(dt), _p(tt)
            if traces is True:
                ht = np.zeros((S, T), np.uint64)
                gt = np.full((S, T + 1), np.nan)
                prm.selhash_trace, prm.dual_trace = _p(ht), _p(gt)
        res = np.zeros(S, RESULT_DTYPE)
        status = esp_solve(self.ctx, prm, res)
        lam = np.zeros((S, P))
        sel = np.zeros((S, J), np.int32)
        dem = np.zeros((S, P), np.int64)
        esp_get_prices(self.ctx, lam)
        esp_get_selection(self.ctx, sel)
        esp_get_demand(self.ctx, dem)
        return Solution(lam, sel, dem, res, status, lt, dt, ht, gt, tt)

    def evaluate(self, lam, mode=ESP_PRICE_NORMALIZED, flags=0):
        S, J, R, P = self.shape
        lam = np.ascontiguousarray(lam, np.float64).reshape(S, P)
        sel = np.zeros((S, J), np.int32)
        dem = np.zeros((S, P), np.int64)
        ms = np.zeros((S, J))
        esp_evaluate(self.ctx, lam, mode, flags, sel, dem, ms)
        return sel, dem, ms

    def launches(self) -> int:
        return esp_last_launch_count(self.ctx)


def plan(job_off: np.ndarray, S: int, J: int, tile_opt: int, max_warps: int):
    """Host tile planner (no GPU): returns (tiles as an n x 8 int32 array, warp_begin)."""
    lib = load_library()
    job_off = np.ascontiguousarray(job_off, np.int64)
    nt, nw = ctypes.c_int32(), ctypes.c_int32()
    st = lib.esp_debug_plan(_p(job_off), S, J, tile_opt, max_warps, None, 0, None, 0, ctypes.byref(nt),
                            ctypes.byref(nw))
    if st not in (ESP_OK, ESP_ERR_OOM):
        raise EspError(st, "esp_debug_plan")
    tiles = np.zeros((max(nt.value, 1), 8), np.int32)
    wb = np.zeros(nw.value + 1, np.int32)
    _check(lib.esp_debug_plan(_p(job_off), S, J, tile_opt, max_warps, _p(tiles), nt.value, _p(wb), nw.value,
                              ctypes.byref(nt), ctypes.byref(nw)), "esp_debug_plan")
    return tiles[:nt.value], wb


def sort_layout(job_off: np.ndarray, S: int, J: int):
    """Sorted layout of a general table (no GPU): (padded offsets, jmap, scen, runk)."""
    lib = load_library()
    job_off = np.ascontiguousarray(job_off, np.int64)
    off = np.zeros(S * J + 1, np.int64)
    jmap, scen, runk = (np.zeros(S * J, np.int32) for _ in range(3))
    _check(lib.esp_debug_sort_layout(_p(job_off), S, J, _p(off), _p(jmap), _p(scen), _p(runk)),
           "esp_debug_sort_layout")
    return off, jmap, scen, runk


def plan_runs(off, scen, runk, S: int, J: int, tile_opt: int, max_warps: int):
    """Host tile planner over a sorted layout (no GPU): (tiles n x 8 int32, warp_begin)."""
    lib = load_library()
    off = np.ascontiguousarray(off, np.int64)
    scen = np.ascontiguousarray(scen, np.int32)
    runk = np.ascontiguousarray(runk, np.int32)
    nt, nw = ctypes.c_int32(), ctypes.c_int32()
    st = lib.esp_debug_plan_runs(_p(off), _p(scen), _p(runk), S, J, tile_opt, max_warps, None, 0, None, 0,
                                 ctypes.byref(nt), ctypes.byref(nw))
    if st not in (ESP_OK, ESP_ERR_OOM):
        raise EspError(st, "esp_debug_plan_runs")
    tiles = np.zeros((max(nt.value, 1), 8), np.int32)
    wb = np.zeros(nw.value + 1, np.int32)
    _check(lib.esp_debug_plan_runs(_p(off), _p(scen), _p(runk), S, J, tile_opt, max_warps, _p(tiles), nt.value,
                                   _p(wb), nw.value, ctypes.byref(nt), ctypes.byref(nw)), "esp_debug_plan_runs")
    return tiles[:nt.value], wb


def esp_debug_set_plan_waves(ctx: int, waves: int) -> None:
    """Warps of the evaluation pass as this many waves of resident CTAs (0: the library's choice)."""
    _check(load_library().esp_debug_set_plan_waves(ctx, waves), "esp_debug_set_plan_waves")


def esp_debug_hold_barrier(ctx: int) -> None:
    """Test hook: the next grid-resident placement solve's barrier never completes, so it ends in
    ESP_ERR_TIMEOUT and poisons the context (see include/esp_debug.h)."""
    _check(load_library().esp_debug_hold_barrier(ctx), "esp_debug_hold_barrier")


def esp_debug_set_pdl(ctx: int, mode: int) -> None:
    """-1 automatic, 0 off, 1 on (programmatic dependent launch of the evaluation passes)."""
    _check(load_library().esp_debug_set_pdl(ctx, mode), "esp_debug_set_pdl")


def esp_debug_set_sorted_layout(ctx: int, enable: bool) -> None:
    _check(load_library().esp_debug_set_sorted_layout(ctx, 1 if enable else 0), "esp_debug_set_sorted_layout")


def esp_debug_set_wait_limit(ctx: int, limit_ms: int) -> None:
    """Limit of a bounded wait of the evaluation passes in ms of the GPU's timer; 0: the default (4 s)."""
    _check(load_library().esp_debug_set_wait_limit(ctx, int(limit_ms)), "esp_debug_set_wait_limit")


def esp_debug_hold_stage(ctx: int) -> None:
    """Test hook: the next solve's first stage never completes, so the solve ends in ESP_ERR_TIMEOUT
    and poisons the context (see include/esp_debug.h)."""
    _check(load_library().esp_debug_hold_stage(ctx), "esp_debug_hold_stage")


def esp_debug_fail_alloc(ctx: int, n: int) -> None:
    """Test hook: the n-th next device allocation of the context fails with ESP_ERR_OOM (n < 0: off)."""
    _check(load_library().esp_debug_fail_alloc(ctx, int(n)), "esp_debug_fail_alloc")


def esp_debug_set_interleave(ctx: int, enable: bool) -> None:
    """Later loads interleave the per-warp pass's table tile by tile (True, the default) or not."""
    _check(load_library().esp_debug_set_interleave(ctx, 1 if enable else 0), "esp_debug_set_interleave")


def esp_debug_set_stage_f32(ctx: int, enable: bool) -> None:
    """Later loads store the units of the tile-interleaved table as fp32 where every unit is below 2^23
    (True, the default) or keep them as integers."""
    _check(load_library().esp_debug_set_stage_f32(ctx, 1 if enable else 0), "esp_debug_set_stage_f32")


def esp_debug_set_persistent(ctx: int, mode: int) -> None:
    """Persistent pass of later solves: -1 automatic (the default), 0 never (one launch per round), 1
    wherever the table can take it."""
    _check(load_library().esp_debug_set_persistent(ctx, int(mode)), "esp_debug_set_persistent")


def esp_debug_persistent(ctx: int) -> int:
    """CTAs of the persistent launch a plain solve of the loaded table uses (0: one launch per round)."""
    g = ctypes.c_int32()
    _check(load_library().esp_debug_persistent(ctx, ctypes.byref(g)), "esp_debug_persistent")
    return g.value


def esp_debug_persist_waits(ctx: int, reset: bool = True):
    """(nanoseconds, number) of the persistent pass's waits for a scenario's prices that had to poll."""
    ns, n = ctypes.c_int64(), ctypes.c_int64()
    _check(load_library().esp_debug_persist_waits(ctx, ctypes.byref(ns), ctypes.byref(n), 1 if reset else 0),
           "esp_debug_persist_waits")
    return ns.value, n.value


def esp_debug_load_profile(ctx: int):
    """(host ms at the seven phase ends of the last load, cudaMalloc calls, cudaFree calls)."""
    ms = (ctypes.c_double * 7)()
    nm, nf = ctypes.c_int64(), ctypes.c_int64()
    _check(load_library().esp_debug_load_profile(ctx, ms, ctypes.byref(nm), ctypes.byref(nf)),
           "esp_debug_load_profile")
    return list(ms), nm.value, nf.value


def esp_debug_pass_kernel(ctx: int) -> int:
    """How the loaded table is evaluated: 0 per-warp pass, two copies per tile; 1 per-warp pass on the
    tile-interleaved table, one copy per tile; 2 factored placement; 3 as 1 with fp32 units."""
    k = ctypes.c_int32()
    _check(load_library().esp_debug_pass_kernel(ctx, ctypes.byref(k)), "esp_debug_pass_kernel")
    return k.value



# --- IAC slowdown predictor (include/esp_iac.h) ------------------------------------------------

def esp_iac_create(device: int = -1, stream: Optional[int] = None) -> int:
    h = ctypes.c_void_p()
    _check(load_library().esp_iac_create(ctypes.byref(h), device, stream), "esp_iac_create")
    return h.value


def esp_iac_set_stream(h: int, stream: Optional[int]) -> None:
    _check(load_library().esp_iac_set_stream(h, stream), "esp_iac_set_stream")


def esp_iac_load_model(h: int, model) -> None:
    """Loads W1, b1, bn1 (4 x H), W2, b2, bn2, W3, b3, eps from any object with those fields."""
    f32 = lambda a: np.ascontiguousarray(a, np.float32)
    W1, b1, bn1, W2, b2, bn2, W3 = (f32(getattr(model, n)) for n in ("W1", "b1", "bn1", "W2", "b2", "bn2", "W3"))
    H = int(W1.shape[0])
    _check(load_library().esp_iac_load_model(h, H, _p(W1), _p(b1), _p(bn1), _p(W2), _p(b2), _p(bn2), _p(W3),
                                             float(model.b3), float(model.eps)), "esp_iac_load_model")


def esp_iac_predict(h: int, rows, pairs, c_mem: float, out) -> None:
    """Device variant: rows (n, 14) fp32, pairs (m, 2) int32 and out (m,) fp32 are CUDA tensors;
    queued on the handle's stream."""
    n_rows = int(rows.shape[0]) if rows is not None else 0
    n_pairs = int(pairs.shape[0]) if pairs is not None else 0
    _check(load_library().esp_iac_predict(h, n_rows, _p(rows), n_pairs, _p(pairs), float(c_mem), _p(out)),
           "esp_iac_predict")


def esp_iac_predict_host(h: int, rows: np.ndarray, pairs: np.ndarray, c_mem: float) -> np.ndarray:
    rows = np.ascontiguousarray(rows, np.float32).reshape(-1, 14)
    pairs = np.ascontiguousarray(pairs, np.int32).reshape(-1, 2)
    out = np.empty(pairs.shape[0], np.float32)
    _check(load_library().esp_iac_predict_host(h, rows.shape[0], _p(rows), pairs.shape[0], _p(pairs), float(c_mem),
                                               _p(out)), "esp_iac_predict_host")
    return out


ESP_IAC_PATH_TENSOR, ESP_IAC_PATH_FMA = 0, 1


def esp_iac_set_path(h: int, path: int) -> None:
    _check(load_library().esp_iac_set_path(h, path), "esp_iac_set_path")


def esp_iac_synchronize(h: int) -> None:
    _check(load_library().esp_iac_synchronize(h), "esp_iac_synchronize")


def esp_iac_debug_set_wait_limit(h: int, limit_ms: int) -> None:
    """Test hook: bound of each wait of the tensor-core kernel for an MMA group (0: the default)."""
    _check(load_library().esp_iac_debug_set_wait_limit(h, int(limit_ms)), "esp_iac_debug_set_wait_limit")


def esp_iac_debug_hold_commit(h: int) -> None:
    """Test hook: the next tensor-path launch leaves one MMA group uncommitted (its wait runs out)."""
    _check(load_library().esp_iac_debug_hold_commit(h), "esp_iac_debug_hold_commit")


def esp_iac_last_launch_count(h: int) -> int:
    n = ctypes.c_int64()
    _check(load_library().esp_iac_last_launch_count(h, ctypes.byref(n)), "esp_iac_last_launch_count")
    return n.value


def esp_iac_destroy(h: int) -> None:
    load_library().esp_iac_destroy(h)


class Predictor:
    """One esp_iac handle: load a model, then predict slowdowns of co-location pairs."""

    def __init__(self, model=None, device: int = -1, stream: Optional[int] = None, path: int = 0):
        self.h = esp_iac_create(device, stream)
        esp_iac_set_path(self.h, path)
        if model is not None:
            esp_iac_load_model(self.h, model)

    def load(self, model) -> None:
        esp_iac_load_model(self.h, model)

    def predict(self, rows, pairs, c_mem: float, out=None):
        """numpy inputs: host call, returns numpy; torch CUDA tensors: device call into `out`."""
        if isinstance(rows, np.ndarray) or isinstance(pairs, np.ndarray):
            return esp_iac_predict_host(self.h, rows, pairs, c_mem)
        esp_iac_predict(self.h, rows, pairs, c_mem, out)
        return out

    def close(self) -> None:
        if self.h:
            esp_iac_destroy(self.h)
            self.h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass
