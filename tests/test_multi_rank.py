"""The multi-GPU host logic of bench.py on CPU with two gloo ranks: each rank owns a disjoint block
of scenarios (weak scaling), the scenarios of the two ranks are different data, and the whole-job
throughput is the sum of the ranks' evaluations over the slowest rank's step time. The per-rank work
here is the oracle on the rank's scenarios (no GPU); the GPU path shards the same way."""

import os
import socket

import numpy as np
import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, out_dir):
    import sys
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    sys.path.insert(0, root)
    import bench
    import oracle
    from paper_2608_07971_gb300 import workloads as W
    dist.init_process_group("gloo", init_method=f"tcp://127.0.0.1:{port}", rank=rank, world_size=world)
    ids = bench.scenario_ids("whatif_batch", rank)
    w = W.whatif_batch(scenarios=ids[:2], J=64)
    t = w.table
    T = 5 + 3 * rank                       # unequal work: the slower rank sets the step time
    import time
    t0 = time.perf_counter()
    sols = oracle.solve(t, w.eta0, T)
    step_s = time.perf_counter() - t0
    evals = t.n_opt * (T + 1)
    value, max_s, total = bench.aggregate(dist, step_s, evals)
    gathered = [None] * world
    dist.all_gather_object(gathered, {"ids": ids, "step_s": step_s, "evals": evals,
                                      "value": value, "max_s": max_s, "total": total,
                                      "first_units": t.units[:4].tolist(), "lam": sols[0].lam.tolist()})
    if rank == 0:
        np.save(os.path.join(out_dir, "gathered.npy"), np.array(gathered, dtype=object), allow_pickle=True)
    dist.barrier()
    dist.destroy_process_group()


def test_two_gloo_ranks_shard_scenarios_and_aggregate(tmp_path):
    port = _free_port()
    mp.start_processes(_rank_main, args=(2, port, str(tmp_path)), nprocs=2, start_method="spawn", join=True)
    g = np.load(tmp_path / "gathered.npy", allow_pickle=True)
    r0, r1 = g[0], g[1]
    assert set(r0["ids"]).isdisjoint(r1["ids"]) and len(r0["ids"]) == len(r1["ids"]) == 1024
    assert r0["ids"][-1] + 1 == r1["ids"][0]                       # contiguous blocks
    assert r0["first_units"] != r1["first_units"]                   # different scenarios, different data
    assert r0["max_s"] == r1["max_s"] == max(r0["step_s"], r1["step_s"])
    assert r0["total"] == r1["total"] == r0["evals"] + r1["evals"]
    assert r0["value"] == pytest.approx((r0["evals"] + r1["evals"]) / max(r0["step_s"], r1["step_s"]))
