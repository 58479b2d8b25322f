#!/usr/bin/env python3
"""Throughput of the ESP tatonnement (Sec. 3.2) on GB300: option-evaluations per second.

One step = one full solve of the workload through the C ABI: T price rounds (each a best response
of every job over every option, the int64 demand sum and the price update of Eq. price_update) and
the final best response, for every scenario of the batch. `value` is measured with the table already
resident in HBM; `e2e` repeats the step through the public API with host inputs (pinned), i.e. the
upload, validation and planning of the table, the solve, and the read-back of selections and prices.

Default workload: heavy_tail (16 scenarios of J=65536 jobs with K_j = min(256, Zipf 1.3) options,
R=6, T=1000: 61.3 M options, 1.96 GB per round), the largest single-GPU configuration; whatif_batch
(1024 independent 512-GPU scenarios, J=2048, K=16, R=6, T=300) is measured beside it as a keyed
second line with its own roofline. Multi-GPU (torchrun): every rank solves its own block of
scenarios (weak scaling, no data-path collective). --impl reference times the oracle (the plain
single-threaded C restatement of the method) instead.
"""

from __future__ import annotations

import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

from paper_2608_07971_gb300 import workloads as W  # noqa: E402

MODE_NAMES = {0: "raw", 1: "normalized"}
STEP_NAMES = {0: "fixed", 1: "inv_sqrt"}
L2_BYTES = 129 * 2**20


def parse_args():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=5)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--workload", default="heavy_tail", choices=sorted(W.WORKLOADS))
    ap.add_argument("--second", default="whatif_batch",
                    help="workload measured beside the main one as a keyed line ('none' to skip)")
    ap.add_argument("--rounds", type=int, default=None, help="override T (changes the workload)")
    ap.add_argument("--scenarios", type=int, default=None, help="override S (profiling of a smaller case)")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-resident", action="store_true", help="skip the cluster-resident measurement")
    ap.add_argument("--no-factored", action="store_true", help="skip the factored placement measurement")
    ap.add_argument("--no-iac", action="store_true", help="skip the IAC predictor measurement")
    ap.add_argument("--iac-scenarios", type=int, default=1024, help="what-if scenarios of the IAC batch")
    ap.add_argument("--cpu-seconds", type=float, default=12.0, help="oracle time budget of the CPU baseline")
    return ap.parse_args()


def rank_info():
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", str(rank)))
    return rank, world, local


def scenario_ids(name: str, rank: int, per=None):
    """Weak scaling: rank r solves its own block of scenarios (same per-rank work)."""
    per = per or {"whatif_batch": 1024, "heavy_tail": 16}.get(name, 1)
    return list(range(rank * per, (rank + 1) * per))


def make_workload(name: str, rank: int, per=None) -> W.Workload:
    return W.make(name, scenarios=scenario_ids(name, rank, per))


def aggregate(dist, step_seconds: float, evals_local: float, device=None):
    """Whole-job throughput under weak scaling: evaluations summed over ranks, divided by the slowest
    rank's step time (max over ranks). dist is torch.distributed or None for one process."""
    if dist is None:
        return evals_local / step_seconds, step_seconds, evals_local
    import torch
    t = torch.tensor([step_seconds], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    e = torch.tensor([float(evals_local)], dtype=torch.float64, device=device)
    dist.all_reduce(e, op=dist.ReduceOp.SUM)
    return float(e.item()) / float(t.item()), float(t.item()), float(e.item())


def config_of(w: W.Workload, T: int) -> dict:
    t = w.table
    K = t.option_counts()
    return {
        "workload": w.name, "S": t.S, "J": t.J, "R": t.R, "P": t.P,
        "K_mean": round(float(K.mean()), 3), "K_max": int(K.max()),
        "rounds": T, "eta0": w.eta0, "price_mode": MODE_NAMES[w.mode], "step": STEP_NAMES[w.step],
        "n_opt": t.n_opt, "table_bytes": t.table_bytes(),
        "l2": "inputs larger than L2 (table %.2f GB vs 129 MB L2)" % (t.table_bytes() / 1e9)
        if t.table_bytes() > L2_BYTES else "table fits in L2 (latency-bound workload)",
        "evals_per_step": t.n_opt * (T + 1),
        "table_sha256": t.digest(),
    }


def measured_peak():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            pk = json.load(f)
        return float(pk["hbm_gbs"]), "measured"
    except Exception:
        return 6800.0, "fallback"


PASS_KERNEL_SOURCES = ("esp_kernels.cu", "esp_kernels_f32.cu", "esp_pass.cuh", "esp_tile.cuh", "esp_ptx.cuh", "esp_warp.cuh", "esp_device.cuh",
                       "esp_common.h", "esp_kernels.h")


def pass_kernel_sha256() -> str:
    """SHA-256 over the sources the evaluation-pass kernel is compiled from, in a fixed order."""
    h = hashlib.sha256()
    for name in PASS_KERNEL_SOURCES:
        with open(os.path.join(ROOT, "paper_2608_07971_gb300", "csrc", name), "rb") as f:
            h.update(f.read())
    return h.hexdigest()


def kernel_traffic(workload: str, n_opt_launch: int):
    """DRAM bytes per evaluation pass from the committed ncu summary of this workload's shape (a
    smaller capture of the same table shape), scaled to this workload's option count, or None when
    there is none or the kernel sources changed since the counters were taken."""
    path = os.path.join(ROOT, "profiles", "pass_traffic.json")
    try:
        with open(path) as f:
            rec = json.load(f)[workload]
        if rec.get("kernel_source_sha256") != pass_kernel_sha256():
            return None
        return float(rec["dram_bytes_per_launch"]) / float(rec["options_per_launch"]) * n_opt_launch
    except Exception:
        return None


# fp32 FMA units of a GB300 (152 SMs x 128 lanes) at the maximum SM clock, 2 flops per FMA
FP32_PEAK_TFLOPS = 152 * 128 * 2 * 2070e6 / 1e12
# nominal dense tf32 / bf16 tensor rate of a GB300 (1.1 / 2.25 PFLOP/s)
TF32_PER_BF16 = 1.1 / 2.25


def tensor_peak_tf32():
    """tf32 tensor peak: the measured bf16 burst peak x the nominal tf32/bf16 ratio."""
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            return float(json.load(f)["bf16_tflops"]) * TF32_PER_BF16, "measured bf16_tflops x nominal tf32/bf16"
    except Exception:
        return 1900.0 * TF32_PER_BF16, "fallback bf16 x nominal tf32/bf16"


def bench_iac(esp, stream, args, dist, barrier):
    """Times esp_iac_predict on the IAC what-if batch (S=1024 scenarios x 2048 jobs x 16
    configurations = 33.5 M pairs, 64 hidden units), one launch per batch: the tensor-core kernel
    (the default) and the CUDA-core kernel beside it."""
    import torch
    from paper_2608_07971_gb300 import workloads as W
    w = W.iac_batch(S=args.iac_scenarios)
    dev = torch.device("cuda", torch.cuda.current_device())
    rows = torch.from_numpy(w.rows).to(dev)
    pairs = torch.from_numpy(w.pairs).to(dev)
    out = torch.empty(len(w.pairs), dtype=torch.float32, device=dev)
    n = len(w.pairs)
    H = w.model.W1.shape[0]

    def timed(path):
        pr = esp.Predictor(w.model, stream=stream.cuda_stream, path=path)
        for _ in range(max(3, args.warmup)):
            pr.predict(rows, pairs, w.c_mem, out)
        esp.esp_iac_synchronize(pr.h)
        barrier()
        torch.cuda.synchronize()
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for _ in range(args.steps):
            pr.predict(rows, pairs, w.c_mem, out)
        e1.record(stream)
        esp.esp_iac_synchronize(pr.h)
        barrier()
        launches = esp.esp_iac_last_launch_count(pr.h)
        pr.close()
        return e0.elapsed_time(e1) / args.steps, launches

    flops = 2 * (36 * H + H * H + H)            # algorithmic flops per pair
    ms_tc, launches = timed(esp.ESP_IAC_PATH_TENSOR)
    ms_fma, _ = timed(esp.ESP_IAC_PATH_FMA)
    value, step_s, _ = aggregate(dist, ms_tc / 1e3, n, device="cuda")
    peak, peak_kind = tensor_peak_tf32()
    achieved = n * flops / (ms_tc / 1e3) / 1e12
    mma_flops = 3 * 2 * (40 * 64 + 64 * 64)      # issued by the split (padded K and N)
    fma_tflops = n * flops / (ms_fma / 1e3) / 1e12
    line = {"value": value, "unit": "pairs/s", "ms_per_step": step_s * 1e3, "pairs_per_step": n,
            "hidden": H, "launches_per_step": launches, "dtype": "f32 (tf32x3 tensor-core products)",
            "roofline": {"bound": "tensor", "kernel": "k_iac_tc (tcgen05 kind::tf32, three-term split)",
                         "achieved": achieved, "peak": peak, "unit": "TFLOP/s", "frac": achieved / peak,
                         "traffic": None, "peak_kind": peak_kind, "flops_per_pair": flops,
                         "mma_flops_per_pair": mma_flops,
                         "tensor_pipe_frac": n * mma_flops / (ms_tc / 1e3) / 1e12 / peak},
            "fma_path": {"ms_per_step": ms_fma, "value": n / (ms_fma / 1e3), "achieved": fma_tflops,
                         "peak": FP32_PEAK_TFLOPS, "unit": "TFLOP/s", "frac": fma_tflops / FP32_PEAK_TFLOPS,
                         "peak_kind": "derived: 152 SMs x 128 fp32 lanes x 2 flops x 2070 MHz"},
            "workload": f"iac_whatif S={w.S} J={w.J} K={w.K}, pair list {w.pairs.nbytes} B (> L2)"}
    del rows, pairs, out
    return line


class ClockSampler:
    """nvidia-smi samples of SM clock and throttle reasons during the timed region."""

    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, uuid=None):
        self.uuid = uuid
        self.proc = None
        self.path = None

    def __enter__(self):
        fd, self.path = tempfile.mkstemp(prefix="clocks_", suffix=".csv")
        os.close(fd)
        cmd = ["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits", "-lms", "200"]
        if self.uuid:
            cmd.insert(1, f"--id={self.uuid}")
        try:
            self.out = open(self.path, "w")
            self.proc = subprocess.Popen(cmd, stdout=self.out, stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None
        return self

    def __exit__(self, *exc):
        if self.proc is not None:
            time.sleep(0.25)
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except Exception:
                self.proc.kill()
            self.out.close()

    def summary(self):
        rows = []
        try:
            for line in open(self.path):
                parts = [p.strip() for p in line.split(",")]
                if len(parts) >= 8:
                    rows.append(parts)
        except Exception:
            pass
        finally:
            try:
                os.unlink(self.path)
            except Exception:
                pass
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unsampled"]}
        sm = [float(r[0]) for r in rows if r[0].replace(".", "").isdigit()]
        mx = [float(r[1]) for r in rows if r[1].replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in rows for i in range(4) if r[4 + i].lower().startswith("active")})
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(mx) if mx else None,
                "reasons": reasons, "samples": len(rows)}


def cpu_baseline(w: W.Workload, T: int, budget_s: float) -> dict:
    """The oracle as it stands, single-threaded, on whole scenarios of the same workload until the
    time budget is spent (at least one scenario; a prefix of its rounds if one scenario alone would
    take more than 2.5 budgets at the rate a short probe measures on this host)."""
    import oracle
    t = w.table
    ot = oracle.OracleTable(t)
    lib = oracle.load()
    per_round = t.n_opt / t.S
    # the oracle's rate on this host, from a few rounds of the first scenario (not counted): a
    # scenario that would take well over the budget runs a prefix of its rounds
    probe = min(T, 4)
    n0 = int(t.job_off[t.J] - t.job_off[0])
    p0 = time.perf_counter()
    oracle.solve_scenario(ot, 0, w.eta0, probe, mode=w.mode, step=w.step, lib=lib)
    s_per_eval = (time.perf_counter() - p0) / max(1, n0 * (probe + 1))
    rounds = T
    if per_round * (T + 1) * s_per_eval > 2.5 * budget_s:
        rounds = max(1, int(budget_s / (per_round * s_per_eval)) - 1)
    evals, n, t0 = 0, 0, time.perf_counter()
    while n < t.S:
        oracle.solve_scenario(ot, n, w.eta0, rounds, mode=w.mode, step=w.step, lib=lib)
        evals += int(t.job_off[(n + 1) * t.J] - t.job_off[n * t.J]) * (rounds + 1)
        n += 1
        if time.perf_counter() - t0 >= budget_s:
            break
    dt = time.perf_counter() - t0
    what = f"{n} of {t.S} scenarios of {w.name}, " + (f"all {T} rounds + final pass" if rounds == T
                                                       else f"first {rounds} rounds + final pass")
    return {"value": evals / dt, "unit": "option-evals/s", "cores": 1, "kind": "oracle",
            "sample": what + f", {dt:.1f} s on 1 of {os.cpu_count()} host cores"}


def run_reference(args):
    rank, world, _ = rank_info()
    if rank != 0:
        return 0
    w = make_workload(args.workload, 0, args.scenarios)
    T = args.rounds if args.rounds is not None else w.rounds
    w.rounds = T
    import oracle
    t = w.table
    ot = oracle.OracleTable(t)
    lib = oracle.load()
    # one step = the oracle's full solve of a fixed number of scenarios, about 1-2 s of CPU work
    t0 = time.perf_counter()
    oracle.solve_scenario(ot, 0, w.eta0, T, mode=w.mode, step=w.step, lib=lib)
    one = time.perf_counter() - t0
    m = int(max(1, min(t.S, round(1.5 / max(one, 1e-6)))))
    rounds = T
    if one > 6.0:       # scenario too large for a step: a prefix of its rounds
        rounds = max(1, int(T * 1.5 / one))
        m = 1

    def step(i):
        for k in range(m):
            s = (i * m + k) % t.S
            oracle.solve_scenario(ot, s, w.eta0, rounds, mode=w.mode, step=w.step, lib=lib)

    for i in range(args.warmup):
        step(i)
    t0 = time.perf_counter()
    for i in range(args.steps):
        step(args.warmup + i)
    dt = (time.perf_counter() - t0) / args.steps
    evals = m * (t.n_opt / t.S) * (rounds + 1)
    value = evals / dt
    sample = f"{m} scenario(s) of {w.name} per step, " + (f"all {T} rounds + final pass" if rounds == T
                                                         else f"first {rounds} rounds + final pass")
    line = {
        "impl": "reference", "metric": "option-evaluations/sec", "value": value, "unit": "option-evals/s",
        "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup, "ms_per_step": dt * 1e3,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic (seeded generator)", "config": config_of(w, T),
        "cpu_baseline": {"value": value, "unit": "option-evals/s", "cores": 1, "kind": "oracle",
                         "sample": sample},
        "e2e": {"value": value, "unit": "option-evals/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)
    return 0


def time_streaming(esp, solver, w, T, args, dist, barrier, stream, clk=None):
    """Times args.steps whole solves of the loaded table (one CUDA graph each, CUDA events on the
    library's stream), then the evaluation passes alone (separate solves with an event pair around
    every pass). Returns the measured line: value, ms per step, roofline of the pass kernel."""
    import torch
    import contextlib
    t = w.table
    ctx = solver.ctx
    prm = solver.params(w.eta0, T, mode=w.mode, step=w.step)
    prm_ev = solver.params(w.eta0, T, mode=w.mode, step=w.step, flags=esp.ESP_FLAG_PASS_EVENTS)
    for _ in range(args.warmup):
        esp.esp_solve_async(ctx, prm)
    stream.synchronize()
    esp.esp_debug_stats(ctx, reset=True)
    launches_per_step = esp.esp_last_launch_count(ctx)
    barrier()
    torch.cuda.synchronize()
    ev0 = torch.cuda.Event(enable_timing=True)
    ev1 = torch.cuda.Event(enable_timing=True)
    with (clk if clk is not None else contextlib.nullcontext()):
        ev0.record(stream)
        for _ in range(args.steps):
            esp.esp_solve_async(ctx, prm)
        ev1.record(stream)
        stream.synchronize()
    torch.cuda.synchronize()
    barrier()
    ms = ev0.elapsed_time(ev1) / args.steps
    res = np.zeros(t.S, esp.RESULT_DTYPE)
    st = esp.esp_get_result(ctx, res)
    assert np.all(res["rounds_run"] == T) or st != 0, "unexpected early stop"
    n_res, n_marked = esp.esp_debug_stats(ctx, reset=True)
    # the pass durations: solves with an event pair around every pass (the last solve's passes)
    for _ in range(2):
        esp.esp_solve_async(ctx, prm_ev)
    stream.synchronize()
    esp.esp_pass_times(ctx, reset=True)
    ev0.record(stream)
    esp.esp_solve_async(ctx, prm_ev)
    ev1.record(stream)
    stream.synchronize()
    ms_ev = ev0.elapsed_time(ev1)
    pass_ms, n_pass = esp.esp_pass_times(ctx, reset=True)

    evals_step = t.n_opt * (T + 1)
    value, step_s, _ = aggregate(dist, ms / 1e3, evals_step, device="cuda")
    peak, peak_kind = measured_peak()
    # the pass's average launch duration in the timed region: the region's time per step over the
    # T + 1 passes of a step (the step's two small kernels, state init and objectives, and the gaps
    # between launches are charged to the passes, so this understates the kernel slightly)
    other_ms = max(0.0, ms_ev - pass_ms)
    avg_ms = max(1e-9, ms / (T + 1))
    bytes_pass = t.table_bytes()
    achieved = bytes_pass / (avg_ms / 1e3) / 1e9
    ev_avg_ms = pass_ms / max(n_pass, 1)
    ev_achieved = bytes_pass / (ev_avg_ms / 1e3) / 1e9 if n_pass else None
    kind = {0: "k_pass (per-warp pass, two bulk copies per tile)",
            1: "k_pass (per-warp pass, one bulk copy per tile from the tile-interleaved table)",
            3: "k_pass (per-warp pass, one bulk copy per tile, fp32 units)"}.get(
        esp.esp_debug_pass_kernel(ctx), "k_place (factored placement pass)")
    persist = esp.esp_debug_persistent(ctx) > 0
    if persist:
        kind = ("k_pass_persist (rounds 0..T-1 in one cooperative launch, scenarios released by their price "
                "updates; one bulk copy per tile, fp32 units) + k_pass (final pass)")
    roofline = {"bound": "hbm", "kernel": kind + ": best response + demand aggregation + fused price update",
                "achieved": achieved, "peak": peak, "unit": "GB/s", "frac": achieved / peak,
                "traffic": kernel_traffic(w.name, t.n_opt),
                "peak_kind": f"{peak_kind} hbm_gbs (copy)",
                "frac_of_nominal_8tbs": achieved / 8000.0,
                "bytes_per_launch": bytes_pass, "avg_launch_ms": avg_ms,
                "launches_per_step": T + 1,
                "persistent": persist,
                "per_round_note": ("the T rounds run in one launch: bytes_per_launch and avg_launch_ms are per "
                                   "round (the step's time over its T + 1 evaluation passes)") if persist else
                                  "one launch per round",
                "event_timed": {"avg_launch_ms": ev_avg_ms, "achieved": ev_achieved,
                                "frac": (ev_achieved / peak) if ev_achieved else None, "launches": n_pass,
                                "ms_per_step_outside_passes": other_ms,
                                "note": "separate solves with an event pair around every pass (each pass then "
                                        "launches alone, without overlapping the kernel before it; per-pass "
                                        "events always use one launch per round)"},
                "exact_resolutions_per_pass": n_res / max(1, (args.warmup + args.steps) * (T + 1)),
                "duplicates_marked": n_marked}
    return {"value": value, "unit": "option-evals/s", "ms_per_step": step_s * 1e3,
            "rounds_per_sec": T / step_s, "evals_per_step": evals_step, "roofline": roofline,
            "launches_per_step": launches_per_step, "device_ms_last_solve": float(res["device_ms"][0])}


def gpu_local_cpus(device: int):
    """The host CPUs on the GPU's own NUMA node (from the PCI device's local_cpulist), or None."""
    try:
        import torch
        p = torch.cuda.get_device_properties(device)
        bus = f"{p.pci_domain_id:04x}:{p.pci_bus_id:02x}:{p.pci_device_id:02x}.0"
        with open(f"/sys/bus/pci/devices/{bus}/local_cpulist") as f:
            spec = f.read().strip()
        cpus = set()
        for part in spec.split(","):
            a, _, b = part.partition("-")
            cpus.update(range(int(a), int(b or a) + 1))
        return cpus or None
    except Exception:
        return None


def time_e2e(esp, solver, w, T, args, dist, barrier, stream, local):
    """The step through the public API from pinned host buffers: every step uploads its table
    (esp_load_options: copy, validation, planning, duplicate marks), solves it, and reads back the
    selections and prices. Two contexts alternate so that step i+1's upload overlaps step i's solve
    (esp_solve_async); every step still pays its own copies, inside the timed region."""
    import torch
    t = w.table
    # the host buffers live on the GPU's own NUMA node: the pinned copies are made (first touched) by
    # this thread while it runs on that node's CPUs
    near = gpu_local_cpus(local)
    numa = "not bound (GPU-local CPUs unknown)"
    if near:
        try:
            os.sched_setaffinity(0, near)
            numa = f"host buffers first touched on the GPU's NUMA node ({len(near)} CPUs)"
        except Exception:
            pass
    pin = lambda a: torch.from_numpy(np.ascontiguousarray(a)).pin_memory()  # noqa: E731
    h_off, h_units, h_vals = pin(t.job_off), pin(t.units), pin(t.values)
    h_grp = None if t.group is None else pin(t.group.view(np.int16))
    h_cap = pin(t.capacity)
    # the upload alone: the host-to-device copy of the step's inputs (a plain torch copy)
    d_probe = torch.empty(h_units.numel() * 4 + h_vals.numel() * 8, dtype=torch.uint8, device="cuda")
    probe = []
    for _ in range(3):
        torch.cuda.synchronize()
        p0 = time.perf_counter()
        d_probe[:h_units.numel() * 4].copy_(h_units.view(torch.uint8).reshape(-1), non_blocking=True)
        d_probe[h_units.numel() * 4:].copy_(h_vals.view(torch.uint8).reshape(-1), non_blocking=True)
        torch.cuda.synchronize()
        probe.append((time.perf_counter() - p0) * 1e3)
    del d_probe
    h_sel = [torch.empty((t.S, t.J), dtype=torch.int32).pin_memory() for _ in range(2)]
    h_lam = [torch.empty((t.S, t.P), dtype=torch.float64).pin_memory() for _ in range(2)]
    # a cold load: a new context (fresh buffers, nothing planned yet), on a stream of its own so that
    # its loads overlap the other context's solves
    torch.cuda.synchronize()
    stream2 = torch.cuda.Stream()
    c0 = time.perf_counter()
    other = esp.Solver(device=local, stream=stream2.cuda_stream)
    esp.esp_load_options(other.ctx, t.S, t.J, t.R, t.P, t.r_global, h_off, h_units, h_vals, h_grp, h_cap)
    torch.cuda.synchronize()
    cold_ms = (time.perf_counter() - c0) * 1e3
    ctxs = [solver.ctx, other.ctx]
    prm = [s.params(w.eta0, T, mode=w.mode, step=w.step) for s in (solver, other)]

    prof = []

    def load(i):
        esp.esp_load_options(ctxs[i], t.S, t.J, t.R, t.P, t.r_global, h_off, h_units, h_vals, h_grp, h_cap)
        prof.append(esp.esp_debug_load_profile(ctxs[i]))

    split = {"load": 0.0, "wait": 0.0}

    def run(steps):
        load(0)
        esp.esp_solve_async(ctxs[0], prm[0])
        for i in range(steps):
            cur, nxt = i % 2, (i + 1) % 2
            c0 = time.perf_counter()
            if i + 1 < steps:
                load(nxt)          # overlaps the current solve
            c1 = time.perf_counter()
            esp.esp_get_selection(ctxs[cur], h_sel[cur])
            esp.esp_get_prices(ctxs[cur], h_lam[cur])
            c2 = time.perf_counter()
            split["load"] += c1 - c0
            split["wait"] += c2 - c1
            if i + 1 < steps:
                esp.esp_solve_async(ctxs[nxt], prm[nxt])

    run(max(2, args.warmup))
    barrier()
    split["load"] = split["wait"] = 0.0
    prof.clear()
    # at least 8 steps: the pipeline's first upload has no solve to hide under
    steps = max(args.steps, 8)
    t0 = time.perf_counter()
    run(steps)
    e2e_s = (time.perf_counter() - t0) / steps
    phases = np.mean([p[0] for p in prof], axis=0).tolist() if prof else None
    allocs = int(sum(p[1] + p[2] for p in prof))
    barrier()
    # a warm load alone (same offsets: the host plan is reused), for the split of a step
    w0 = time.perf_counter()
    load(1)
    warm_ms = (time.perf_counter() - w0) * 1e3
    evals_step = t.n_opt * (T + 1)
    e2e_value, e2e_s, _ = aggregate(dist, e2e_s, evals_step, device="cuda")
    h2d = t.job_off.nbytes + t.units.nbytes + t.values.nbytes + t.capacity.nbytes + \
        (0 if t.group is None else t.group.nbytes)
    d2h = h_sel[0].numel() * 4 + h_lam[0].numel() * 8
    other.close()
    return {"value": e2e_value, "unit": "option-evals/s", "h2d_bytes_per_step": int(h2d),
            "d2h_bytes_per_step": int(d2h), "ms_per_step": e2e_s * 1e3,
            "cold_load_ms": cold_ms, "warm_load_ms": warm_ms, "upload_alone_ms": probe,
            "steps": steps,
            "split_ms_per_step": {"load_overlapping_solve": split["load"] * 1e3 / steps,
                                  "wait_for_solve_and_read_back": split["wait"] * 1e3 / steps},
            "load_profile_ms": {"uploads_validation_queued": phases[0], "sorted_layout_queued": phases[1],
                                "occupancy": phases[2], "planned": phases[3], "validated_marked": phases[4],
                                "state_queued": phases[5], "returned": phases[6],
                                "cuda_malloc_free_calls": allocs} if phases else None,
            "pipeline": "two contexts: step i+1's upload overlaps step i's solve", "host_memory": numa}


def run_ours(args):
    import torch
    rank, world, local = rank_info()
    if not torch.cuda.is_available():
        raise SystemExit("bench.py needs a CUDA GPU (no CPU fallback)")
    torch.cuda.set_device(local)
    dist = None
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))

    from paper_2608_07971_gb300 import build, esp
    if not os.path.exists(esp.LIB_PATH):
        build.build()
    esp.load_library()

    def barrier():
        if dist is not None:
            dist.barrier()

    w = make_workload(args.workload, rank, args.scenarios)
    T = args.rounds if args.rounds is not None else w.rounds
    t = w.table
    stream = torch.cuda.Stream()
    solver = esp.Solver(t, device=local, stream=stream.cuda_stream)
    ctx = solver.ctx

    uuid = None
    try:
        uuid = str(torch.cuda.get_device_properties(local).uuid)
        if uuid and not uuid.startswith("GPU-"):
            uuid = "GPU-" + uuid
    except Exception:
        uuid = None

    clk = ClockSampler(uuid)
    main = time_streaming(esp, solver, w, T, args, dist, barrier, stream, clk)
    value, ms_max = main["value"], main["ms_per_step"]

    # the cluster-resident path (all rounds in one launch, tables in shared memory) on the same
    # workload, when the table qualifies: a second measured line beside the streaming one
    resident = None
    shape = esp.esp_debug_resident(ctx) if not args.no_resident else None
    if shape is not None:
        lam_stream = np.zeros((t.S, t.P))
        esp.esp_get_prices(ctx, lam_stream)
        prm_res = solver.params(w.eta0, T, mode=w.mode, step=w.step, flags=esp.ESP_FLAG_RESIDENT)
        for _ in range(args.warmup):
            esp.esp_solve_async(ctx, prm_res)
        barrier()
        torch.cuda.synchronize()
        r0 = torch.cuda.Event(enable_timing=True)
        r1 = torch.cuda.Event(enable_timing=True)
        r0.record(stream)
        for _ in range(args.steps):
            esp.esp_solve_async(ctx, prm_res)
        r1.record(stream)
        stream.synchronize()
        barrier()
        res_ms = r0.elapsed_time(r1) / args.steps
        res_value, res_s, _ = aggregate(dist, res_ms / 1e3, t.n_opt * (T + 1), device="cuda")
        lam_res = np.zeros((t.S, t.P))
        esp.esp_get_prices(ctx, lam_res)
        resident = {"value": res_value, "unit": "option-evals/s", "ms_per_step": res_s * 1e3,
                    "rounds_per_sec": T / res_s, "cluster_ctas": shape[0], "clusters_co_resident": shape[1],
                    "launches_per_step": esp.esp_last_launch_count(ctx),
                    "same_prices_as_streaming": bool(np.array_equal(lam_res, lam_stream)),
                    "note": "ESP_FLAG_RESIDENT: each scenario's table read from HBM once per solve, then held "
                            "in the shared memory of one thread-block cluster for all rounds (the library "
                            "falls back to streaming where its cost model predicts the resident solve slower)"}

    # the factored placement path (configurations x nodes computed on the fly, esp_load_placement)
    factored = None
    if w.factors is not None and not args.no_factored:
        factored = bench_factored(esp, w, T, args, dist, barrier, stream, local, ctx)

    # the IAC slowdown predictor (Eq. dnn_pred) over the what-if batch's co-location pairs
    iac_line = None if args.no_iac else bench_iac(esp, stream, args, dist, barrier)

    # end to end through the public API with host inputs
    e2e = None if args.no_e2e else time_e2e(esp, solver, w, T, args, dist, barrier, stream, local)
    solver.close()

    # the second batched workload, measured the same way, as a keyed line
    second = None
    if args.second != "none" and args.second != args.workload and args.scenarios is None and args.rounds is None:
        w2 = make_workload(args.second, rank)
        s2 = esp.Solver(w2.table, device=local, stream=stream.cuda_stream)
        second = time_streaming(esp, s2, w2, w2.rounds, args, dist, barrier, stream)
        second["config"] = config_of(w2, w2.rounds)
        s2.close()
        del w2, s2

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        cpu = cpu_baseline(w, T, args.cpu_seconds)

    clocks = clk.summary()
    line = {
        "metric": "option-evaluations/sec", "value": value, "unit": "option-evals/s",
        "n_gpus": world, "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms_max,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic (seeded generator, shapes of the named workload)",
        "config": config_of(w, T),
        "run": {"parallelism": f"scenarios sharded over {world} GPU(s), no collective",
                "launch": "one CUDA graph per solve: T+3 launches; pass durations from separate solves with an "
                          "event pair around every pass"},
        "rounds_per_sec": main["rounds_per_sec"],
        "roofline": main["roofline"],
        "device_ms_last_solve": main["device_ms_last_solve"],
        "cpu_baseline": cpu,
        "e2e": e2e,
        args.second if second is not None else "second": second,
        "resident": resident,
        "factored": factored,
        "iac": iac_line,
        "clocks": {k: clocks.get(k) for k in ("sm_mhz", "sm_max_mhz", "reasons")},
        "gpu_launches": int(main["launches_per_step"] * args.steps),
    }
    if rank == 0:
        print(json.dumps(line), flush=True)
    if dist is not None:
        dist.destroy_process_group()
    return 0


def bench_factored(esp, w, T, args, dist, barrier, stream, local, ctx):
    """esp_load_placement on the placement workload: per-round launches and the grid-resident solve."""
    import torch
    t = w.table
    evals_step = t.n_opt * (T + 1)
    lam_stream = np.zeros((t.S, t.P))
    esp.esp_get_prices(ctx, lam_stream)
    fs = esp.Solver(device=local, stream=stream.cuda_stream)
    fs.load_placement(w.factors)

    def timed(flags):
        prm_f = fs.params(w.eta0, T, mode=w.mode, step=w.step, flags=flags)
        for _ in range(args.warmup):
            esp.esp_solve_async(fs.ctx, prm_f)
        barrier()
        torch.cuda.synchronize()
        f0 = torch.cuda.Event(enable_timing=True)
        f1 = torch.cuda.Event(enable_timing=True)
        f0.record(stream)
        for _ in range(args.steps):
            esp.esp_solve_async(fs.ctx, prm_f)
        f1.record(stream)
        stream.synchronize()
        barrier()
        f_ms = f0.elapsed_time(f1) / args.steps
        f_value, f_s, _ = aggregate(dist, f_ms / 1e3, evals_step, device="cuda")
        lam_f = np.zeros((t.S, t.P))
        esp.esp_get_prices(fs.ctx, lam_f)
        return f_value, f_s, esp.esp_last_launch_count(fs.ctx), bool(np.array_equal(lam_f, lam_stream))

    f_value, f_s, f_launches, same_f = timed(0)
    fr_value, fr_s, fr_launches, same_fr = timed(esp.ESP_FLAG_RESIDENT)
    f = w.factors
    fbytes = f.cfg_units.nbytes + f.cfg_values.nbytes + f.sens.nbytes + f.job_type.nbytes
    fs.close()
    return {"value": f_value, "unit": "option-evals/s", "ms_per_step": f_s * 1e3,
            "rounds_per_sec": T / f_s, "bytes_per_pass": int(fbytes), "launches_per_step": f_launches,
            "same_prices_as_streaming": same_f,
            "grid_resident": {"value": fr_value, "ms_per_step": fr_s * 1e3, "rounds_per_sec": T / fr_s,
                              "launches_per_step": fr_launches, "same_prices_as_streaming": same_fr},
            "note": "esp_load_placement: configurations x nodes scored from the factors, the expanded "
                    "options are never stored; evaluations counted over the expanded options; "
                    "grid_resident = ESP_FLAG_RESIDENT, every round in one cooperative launch"}


def main():
    args = parse_args()
    if args.impl == "reference":
        return run_reference(args)
    return run_ours(args)


if __name__ == "__main__":
    sys.exit(main())
