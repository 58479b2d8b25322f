"""Mutation sweep of the host tile planner (test infrastructure, run by hand; a few minutes on all cores).

The library checks every plan before a launch (check_plan in csrc/esp_plan.cpp) and refuses the
table when the check fails. This sweep asks whether that check is complete. Every single-token
change of a comparison, an addition or subtraction, a +-1 offset, an equality test or a logical
and is planted in a temporary copy of csrc/esp_plan.cpp. Each copy is built into
tests/host_sanitized_driver.cpp (without sanitizers) and run on the planner cases of
tests/test_host_sanitized.py. Each outcome is classified:
  - rejected: the planner's own check refused a plan (the driver exits with status 3);
  - crashed: the driver did not finish (the load would fail or fault);
  - valid: every plan still covers every job exactly once, in order, within its tile and warp
    limits (the independent checker of tests/test_abi_host.py);
  - INVALID PLAN ACCEPTED: a plan passed check_plan and failed the independent checker, which
    would be a gap in the library's check. The sweep prints these, and there should be none.

    python -m tests.planner_mutation_sweep
"""

from __future__ import annotations

import concurrent.futures as cf
import os
import shutil
import subprocess
import sys
import tempfile

import numpy as np

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
CSRC = os.path.join(ROOT, "paper_2608_07971_gb300", "csrc")
OPS = [(" < ", " <= "), (" <= ", " < "), (" > ", " >= "), (" >= ", " > "), (" + ", " - "), (" - ", " + "),
       ("+ 1", "+ 2"), ("- 1", "- 2"), (" == ", " != "), ("&&", "||")]


def candidates(lines):
    for i, ln in enumerate(lines):
        if not ln.strip() or ln.strip().startswith("//"):
            continue
        code = ln.split("//")[0]
        for a, b in OPS:
            at = code.find(a)
            while at >= 0:
                yield i, ln[:at] + b + ln[at + len(a):]
                at = code.find(a, at + 1)


def covers(off, tiles6, wb, tile_opt, warps):
    """The tiles walk the (possibly sorted) table once, in order: each starts where the previous one
    ended; a whole-job tile starts and ends on job boundaries; a chunk stays inside one job; no tile
    exceeds tile_opt options; warp ranges are contiguous and within the warp limit. The scenario of
    a tile is not checked here (a sorted layout interleaves the scenarios' runs); for the plain
    layout the independent checker of tests/test_abi_host.py checks it."""
    n_jobs = len(off) - 1
    pos, job = int(off[0]), 0
    for ob, jb, n_opt, n_job, _, flags in tiles6:
        if not 1 <= n_opt <= tile_opt or ob != pos or jb != job:
            return False
        if flags & 1:                                   # a chunk of a large job
            if ob + n_opt > off[jb + 1]:
                return False
            pos = ob + n_opt
            job += int(pos == off[jb + 1])
        else:
            if n_job < 1 or jb + n_job > n_jobs or ob != off[jb] or ob + n_opt != off[jb + n_job]:
                return False
            pos, job = int(off[jb + n_job]), jb + n_job
    return (pos == off[-1] and job == n_jobs and wb[0] == 0 and wb[-1] == len(tiles6)
            and bool(np.all(np.diff(wb) >= 0)) and len(wb) - 1 <= warps)


def plans_valid(out_path, cases):
    """True when every tile plan in the driver's output covers its table."""
    from tests import test_abi_host as abi
    from tests import test_host_sanitized as san
    wd = san._Words(np.fromfile(out_path, np.int64))
    try:
        for S, J, tile_opt, warps, cs, off in cases:
            off = np.asarray(off, np.int64)
            plan = san._read_plan(wd)
            if plan is not None:
                tiles6, wb = plan
                t8 = np.zeros((len(tiles6), 8), np.int64)
                t8[:, 0], t8[:, 1] = tiles6[:, 0] & 0xFFFFFFFF, tiles6[:, 0] >> 32
                t8[:, 2], t8[:, 3] = tiles6[:, 1] & 0xFFFFFFFF, tiles6[:, 1] >> 32
                t8[:, 4:8] = tiles6[:, 2:6]
                abi.tiles_cover(off, S, J, t8, wb, tile_opt)
                if not covers(off, tiles6, wb, tile_opt, warps):
                    return False
            if wd.take():
                n = S * J
                soff = wd.take(n + 1)
                wd.take(n), wd.take(n), wd.take(n)
                splan = san._read_plan(wd)
                if splan is not None and not covers(soff, splan[0], splan[1], tile_opt, warps):
                    return False
            if wd.take():
                wd.take(), wd.take()
                wd.take(wd.take())
    except (AssertionError, IndexError, ValueError):
        return False
    return True


def run_one(n, i, mutated, lines, tmp, cases_bin, cases):
    d = os.path.join(tmp, f"m{n}")
    os.makedirs(d)
    src = os.path.join(d, "esp_plan.cpp")
    open(src, "w").write("\n".join(lines[:i] + [mutated] + lines[i + 1:]))
    exe = os.path.join(d, "driver")
    if subprocess.run(["g++", "-std=c++17", "-O1", "-I", os.path.join(ROOT, "include"), "-I", CSRC,
                       os.path.join(ROOT, "tests", "host_sanitized_driver.cpp"), src,
                       os.path.join(CSRC, "esp_host.cpp"), "-o", exe], capture_output=True).returncode:
        return "build failed", i, mutated
    try:
        r = subprocess.run([exe, cases_bin, os.path.join(d, "out.bin")], capture_output=True, timeout=120)
    except subprocess.TimeoutExpired:
        return "crashed", i, mutated
    if r.returncode == 3:
        return "rejected", i, mutated
    if r.returncode != 0:
        return "crashed", i, mutated
    return ("valid" if plans_valid(os.path.join(d, "out.bin"), cases) else "INVALID PLAN ACCEPTED"), i, mutated


def main() -> int:
    sys.path.insert(0, ROOT)
    from tests import test_host_sanitized as san
    lines = open(os.path.join(CSRC, "esp_plan.cpp")).read().split("\n")
    cases, host = san.host_cases()
    tmp = tempfile.mkdtemp()
    cases_bin = os.path.join(tmp, "cases.bin")
    san._encode(cases, host).tofile(cases_bin)
    counts = {}
    with cf.ThreadPoolExecutor(max_workers=os.cpu_count() or 4) as ex:
        futs = [ex.submit(run_one, n, i, m, lines, tmp, cases_bin, cases) for n, (i, m) in enumerate(candidates(lines))]
        for f in cf.as_completed(futs):
            kind, i, mutated = f.result()
            counts[kind] = counts.get(kind, 0) + 1
            if kind == "INVALID PLAN ACCEPTED":
                print(f"{kind}: line {i + 1}: {lines[i].strip()}  =>  {mutated.strip()}", flush=True)
    shutil.rmtree(tmp, ignore_errors=True)
    print(counts)
    return 0


if __name__ == "__main__":
    sys.exit(main())
