"""Host code under AddressSanitizer and UndefinedBehaviorSanitizer (no GPU).

- The C oracle, built with both sanitizers, passes every pin and gives the plain build's outputs bit
  for bit on the workload shapes and on ragged random tables (run in a child process with the
  sanitizer runtime preloaded, since the interpreter itself is not instrumented).
- The library's host planners (tile plan, sorted layout, cluster-resident slices) and host formulas
  (adaptive threshold, effective capacity), built with both sanitizers into a test driver, accept and
  reject the same tables as the plain library and return the same plans; the resident slices are
  checked against the rule restated here.
- Each harness is shown to be live: a heap overflow and a signed overflow planted in temporary
  copies of the oracle are reported.
"""

import os
import shutil
import subprocess
import sys

import numpy as np
import pytest

import oracle
from paper_2608_07971_gb300 import esp, workloads as W
from tests import sanitized_oracle_run as run

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
CSRC = os.path.join(ROOT, "paper_2608_07971_gb300", "csrc")
SAN = ["-g", "-fsanitize=address,undefined,float-cast-overflow", "-fno-sanitize-recover=all",
       "-fno-omit-frame-pointer"]
SAN_ENV = {"ASAN_OPTIONS": "detect_leaks=0:abort_on_error=0:exitcode=23",
           "UBSAN_OPTIONS": "print_stacktrace=1:halt_on_error=1:exitcode=24"}


def _runtime(name):
    path = subprocess.run(["gcc", f"-print-file-name={name}"], capture_output=True, text=True).stdout.strip()
    return path if os.path.isabs(path) and os.path.exists(path) else None


@pytest.fixture(scope="module")
def asan_rt(tmp_path_factory):
    rt = _runtime("libasan.so")
    if rt is None:
        pytest.skip("gcc has no AddressSanitizer runtime")
    d = tmp_path_factory.mktemp("probe")
    probe = d / "p.c"
    probe.write_text("int main(void) { return 0; }\n")
    if subprocess.run(["gcc", *SAN, str(probe), "-o", str(d / "p")], capture_output=True).returncode != 0:
        pytest.skip("gcc cannot link with the sanitizers")
    return rt


def build_oracle(src_dir, out, replace=None):
    """The oracle (optionally with one planted change) built with both sanitizers."""
    src = open(os.path.join(os.path.dirname(oracle.__file__), "esp_oracle.c")).read()
    if replace:
        assert src.count(replace[0]) == 1, "planted-change anchor missing"
        src = src.replace(*replace)
    c = os.path.join(src_dir, "esp_oracle.c")
    open(c, "w").write(src)
    shutil.copy(os.path.join(os.path.dirname(oracle.__file__), "esp_oracle.h"), src_dir)
    subprocess.check_call(["gcc", *oracle.CFLAGS, *SAN, c, "-o", str(out), "-lm"])
    return str(out)


def run_child(rt, lib, out, pins=False):
    env = dict(os.environ, LD_PRELOAD=rt, **SAN_ENV)
    cmd = [sys.executable, "-m", "tests.sanitized_oracle_run", lib, str(out)] + (["--pins"] if pins else [])
    return subprocess.run(cmd, cwd=ROOT, env=env, capture_output=True, text=True, timeout=600)


def test_oracle_under_sanitizers_matches_plain_build(asan_rt, tmp_path):
    lib = build_oracle(str(tmp_path), tmp_path / "liboracle_san.so")
    r = run_child(asan_rt, lib, tmp_path / "san.npz", pins=True)
    assert r.returncode == 0, r.stderr[-4000:]
    assert "runtime error" not in r.stderr and "Sanitizer" not in r.stderr, r.stderr[-4000:]
    got = np.load(tmp_path / "san.npz")
    want = run.run_cases(oracle.load())
    assert set(got.files) == set(want)
    for k, v in want.items():
        assert np.array_equal(got[k], v, equal_nan=v.dtype.kind == "f"), k


@pytest.mark.parametrize("plant", [
    # a scratch buffer one element short: effective prices write past its end
    ("double *p = (double *)malloc(sizeof(double) * (size_t)t->P);\n    esp_oracle_effective_prices",
     "double *p = (double *)malloc(sizeof(double) * (size_t)(t->P - 1));\n    esp_oracle_effective_prices",
     "heap-buffer-overflow"),
    # the group stride scaled past int32 for every grouped option
    ("(t->R - t->r_global) * (int32_t)t->group[o]", "(t->R - t->r_global) * (int32_t)t->group[o] * 0x40000000",
     "signed integer overflow"),
])
def test_sanitizers_report_planted_mistakes(asan_rt, tmp_path, plant):
    old, new, report = plant
    lib = build_oracle(str(tmp_path), tmp_path / "liboracle_planted.so", (old, new))
    r = run_child(asan_rt, lib, tmp_path / "planted.npz")
    assert r.returncode != 0
    assert report in r.stderr, r.stderr[-2000:]


# ---- the library's host code ----

def _encode(cases, host):
    w = [len(cases)]
    for S, J, tile_opt, warps, cs, off in cases:
        w += [S, J, tile_opt, warps, cs, *np.asarray(off, np.int64).tolist()]
    f64 = lambda x: int(np.array([x], np.float64).view(np.int64)[0])
    tau_base, beta, util, target, beta_max, cap, q_off, q_units, gamma = host
    w += [len(tau_base), *[f64(x) for x in tau_base], f64(beta), f64(util), f64(target), f64(beta_max)]
    w += [len(cap), *cap.tolist(), len(q_off) - 1, *q_off.tolist(), *q_units.ravel().tolist(), f64(gamma)]
    return np.array(w, np.int64)


class _Words:
    def __init__(self, a):
        self.a, self.i = a, 0

    def take(self, n=None):
        if n is None:
            self.i += 1
            return int(self.a[self.i - 1])
        self.i += n
        return self.a[self.i - n:self.i]


def _plan_fields(tiles):
    """esp_debug_plan's 8-int32 tile rows as (opt_begin, job_begin, n_opt, n_job, scenario, flags)."""
    t = tiles.astype(np.int64)
    ob = (t[:, 0] & 0xFFFFFFFF) | (t[:, 1] << 32)
    jb = (t[:, 2] & 0xFFFFFFFF) | (t[:, 3] << 32)
    return np.stack([ob, jb, t[:, 4], t[:, 5], t[:, 6], t[:, 7] & 0xFFFFFFFF], axis=1)


def _read_plan(wd):
    if not wd.take():
        return None
    nt, nw = wd.take(), wd.take()
    return wd.take(6 * nt).reshape(nt, 6), wd.take(nw + 1)


def resident_cuts(off, S, J, cs):
    """Slices of every scenario into cs runs of about equal option counts: run c starts at the first
    job whose first option lies at least floor(c * N_s / cs) options into the scenario."""
    cuts = np.zeros((S, cs + 1), np.int64)
    m_max = n_max = 0
    for s in range(S):
        o = off[s * J:(s + 1) * J + 1]
        N = int(o[J] - o[0])
        cuts[s, cs] = J
        for c in range(1, cs):
            j = int(np.searchsorted(o[:J], o[0] + (N * c) // cs, side="left"))
            cuts[s, c] = max(j, cuts[s, c - 1])
        m_max = max(m_max, int(np.diff(cuts[s]).max()))
        n_max = max(n_max, int(np.diff(o[cuts[s]]).max()))
    return cuts.ravel(), m_max, n_max


def host_cases():
    rng = np.random.default_rng(41)
    tables = [W.tiny_cluster().table, W.whatif_batch(scenarios=[0, 3, 7], J=512).table,
              W.heavy_tail(scenarios=[0], J=16384).table, W.placement_expanded(scenarios=[0], J=64).table,
              W.cluster_512(scenarios=[0, 1], J=2048).table]
    offs = [(t.S, t.J, t.job_off, esp.load_library().esp_debug_tile_options(t.R, int(t.group is not None))) for t in tables]
    for S, J, K in ((3, 500, rng.integers(1, 300, 1500)), (2, 40, rng.choice([1, 2, 700, 1500], 80)),
                    (1, 1, np.array([1])), (5, 1, np.array([3, 1, 77, 2, 129])), (2, 64, np.full(128, 2))):
        off = np.zeros(S * J + 1, np.int64)
        off[1:] = np.cumsum(K)
        offs.append((S, J, off, 128))
    cases = []
    for i, (S, J, off, tile_opt) in enumerate(offs):
        for warps, cs in ((1, 1), (7, 2), (4864, 8), (100000, 16)):
            cases.append((S, J, tile_opt if i % 2 == 0 else 32, warps, cs, off))
    bad = np.array([0, 4, 3, 9], np.int64)             # a job with a negative option count
    cases.append((1, 3, 128, 8, 2, bad))
    cases.append((1, 3, 128, 8, 2, np.array([0, 4, 4, 9], np.int64)))   # a job without options
    cases.append((1, 3, 40, 8, 2, np.array([0, 4, 5, 9], np.int64)))    # tile size not a multiple of 32
    K = rng.integers(1, 5, 25)
    q_off = np.zeros(26, np.int64)
    q_off[1:] = np.cumsum(K)
    host = (rng.random(40) + 1.0, 0.3, 0.93, 0.8, 0.05, np.array([40000, 1 << 53, 9000], np.int64), q_off,
            rng.integers(0, 1000, (int(q_off[-1]), 3)).astype(np.int32), 0.37)
    return cases, host


@pytest.fixture(scope="module")
def host_driver(asan_rt, tmp_path_factory):
    from paper_2608_07971_gb300 import build
    build.build()
    esp.load_library()
    d = tmp_path_factory.mktemp("driver")
    exe = d / "host_driver"
    subprocess.check_call(["g++", "-std=c++17", "-O1", "-ffp-contract=off", *SAN, "-I", os.path.join(ROOT, "include"),
                           "-I", CSRC, os.path.join(ROOT, "tests", "host_sanitized_driver.cpp"),
                           os.path.join(CSRC, "esp_plan.cpp"), os.path.join(CSRC, "esp_host.cpp"), "-o", str(exe)])
    return exe


def test_host_planners_under_sanitizers_match_library(host_driver, tmp_path):
    cases, host = host_cases()
    _encode(cases, host).tofile(tmp_path / "cases.bin")
    r = subprocess.run([str(host_driver), str(tmp_path / "cases.bin"), str(tmp_path / "out.bin")],
                       env=dict(os.environ, **SAN_ENV), capture_output=True, text=True, timeout=600)
    assert r.returncode == 0, r.stderr[-4000:]
    wd = _Words(np.fromfile(tmp_path / "out.bin", np.int64))
    n_ok = 0
    for S, J, tile_opt, warps, cs, off in cases:
        plan = _read_plan(wd)
        try:
            tiles, wb = esp.plan(off, S, J, tile_opt, warps)
        except esp.EspError:
            assert plan is None
        else:
            assert plan is not None
            assert np.array_equal(plan[0], _plan_fields(tiles)) and np.array_equal(plan[1], wb)
            n_ok += 1
        if wd.take():
            n = S * J
            got = [wd.take(n + 1), wd.take(n), wd.take(n), wd.take(n)]
            for a, b in zip(got, esp.sort_layout(off, S, J)):
                assert np.array_equal(a, b)
            runs = _read_plan(wd)
            try:
                tiles, wb = esp.plan_runs(got[0], got[2], got[3], S, J, tile_opt, warps)
            except esp.EspError:
                assert runs is None
            else:
                assert np.array_equal(runs[0], _plan_fields(tiles)) and np.array_equal(runs[1], wb)
        else:
            with pytest.raises(esp.EspError):
                esp.sort_layout(off, S, J)
        valid = off[0] == 0 and np.all(np.diff(off) >= 1)
        if wd.take():
            m_max, n_max = wd.take(), wd.take()
            n_cuts = wd.take()
            assert n_cuts == S * (cs + 1)
            got = wd.take(n_cuts)
            if valid:   # on rejected tables the slices are never used; the sanitizers still watch them
                cuts, m_want, n_want = resident_cuts(off, S, J, cs)
                assert np.array_equal(got, cuts) and (m_max, n_max) == (m_want, n_want)
        else:
            assert not valid
    assert n_ok >= 4 * 10
    tau_base, beta, util, target, beta_max, cap, q_off, q_units, gamma = host
    assert wd.take() == esp.ESP_OK
    tau = wd.take(len(tau_base)).view(np.float64)
    assert np.array_equal(tau, esp.esp_adaptive_threshold(tau_base, beta, util, target, beta_max))
    assert wd.take() == esp.ESP_OK
    assert np.array_equal(wd.take(len(cap)), esp.esp_effective_capacity(cap, q_off, q_units, gamma))
    assert wd.i == len(wd.a)


def test_capacity_range_check_prevents_float_cast_overflow(asan_rt, tmp_path):
    """Without the capacity range check of esp_effective_capacity, a capacity of 2^63 - 1 rounds to
    2^63 in fp64 and its floor no longer fits int64: the sanitized driver reports the conversion."""
    src = open(os.path.join(CSRC, "esp_host.cpp")).read()
    check = "        if (capacity[r] < 1 || capacity[r] > kMaxCapacity)\n            return ESP_ERR_INVALID_ARG;\n"
    assert src.count(check) == 1
    (tmp_path / "esp_host.cpp").write_text(src.replace(check, ""))
    exe = tmp_path / "driver_planted"
    subprocess.check_call(["g++", "-std=c++17", "-O1", "-ffp-contract=off", *SAN, "-I", os.path.join(ROOT, "include"),
                           "-I", CSRC, os.path.join(ROOT, "tests", "host_sanitized_driver.cpp"),
                           os.path.join(CSRC, "esp_plan.cpp"), str(tmp_path / "esp_host.cpp"), "-o", str(exe)])
    q_off = np.array([0, 1], np.int64)
    host = (np.ones(2), 0.3, 0.9, 0.8, 0.1, np.array([np.iinfo(np.int64).max], np.int64), q_off,
            np.zeros((1, 1), np.int32), 0.0)
    _encode([], host).tofile(tmp_path / "cases.bin")
    r = subprocess.run([str(exe), str(tmp_path / "cases.bin"), str(tmp_path / "out.bin")],
                       env=dict(os.environ, **SAN_ENV), capture_output=True, text=True, timeout=300)
    assert r.returncode != 0
    assert "outside the range of representable values" in r.stderr, r.stderr[-2000:]
