"""The streaming pass's host planner (no GPU), checked against its rules restated here.

Blocks: whole jobs of one run and scenario, as many whole rows as fit a stage (a row: K >= 4:
32 / 2^ceil(log2(K/4)) jobs, one job above 128 options; K < 4: 128 / K jobs), covering every job once
and in order; a block is shorter only where its run or scenario ends. CTAs: contiguous block ranges
covering every block, balanced by bytes. Arrivals: a scenario's price update waits until all of its
blocks are counted in (each consumer warp adds the blocks it evaluated), so the target is the
scenario's block count: a wrong count would update too early or never.
"""

import numpy as np
import pytest

from paper_2608_07971_gb300 import esp, workloads as W


@pytest.fixture(scope="module", autouse=True)
def lib():
    from paper_2608_07971_gb300 import build
    build.build()
    return esp.load_library()


def row_jobs(K):
    if K < 4:
        return 128 // K
    m = K // 4
    if m > 32:
        return 1
    lanes = 1
    while lanes < m:
        lanes *= 2
    return 32 // lanes


def block_jobs(K, stage_opt):
    row = row_jobs(K)
    return min(row * max(1, stage_opt // (row * K)), stage_opt // K)


def check(plan, off, S, J, scen, runk, K_uniform):
    tiles, cta, arr, so = plan["tiles"], plan["cta_begin"], plan["arrivals"], plan["stage_opt"]
    n_jobs = S * J
    jscen = scen if scen is not None else np.arange(n_jobs) // J
    jk = runk if runk is not None else np.full(n_jobs, K_uniform)
    nxt = 0
    for t in tiles:
        opt, job = int(t[0]) | (int(t[1]) << 32), int(t[2]) | (int(t[3]) << 32)
        n_opt, n_job, s, fl = int(t[4]), int(t[5]), int(t[6]), int(t[7]) & 0xffffffff
        K = (fl >> 8) & 0xFFF
        assert fl & 8 and job == nxt and 1 <= n_job <= block_jobs(K, so) and n_opt <= so
        assert opt == off[job] and n_opt == K * n_job == off[job + n_job] - off[job]
        assert np.all(jscen[job:job + n_job] == s) and np.all(jk[job:job + n_job] == K)
        if K >= 4:
            assert opt % 4 == 0
        # a block is as long as its stage allows, unless the run or scenario ends
        if n_job < block_jobs(K, so) and job + n_job < n_jobs:
            assert jscen[job + n_job] != s or jk[job + n_job] != K
        nxt = job + n_job
    assert nxt == n_jobs
    assert cta[0] == 0 and cta[-1] == len(tiles) and np.all(np.diff(cta) >= 0)
    assert np.array_equal(arr, np.bincount(tiles[:, 6], minlength=S))
    assert np.all(arr[np.unique(jscen)] >= 1)


@pytest.mark.parametrize("K", [1, 2, 4, 8, 16, 32])
@pytest.mark.parametrize("R", [4, 6, 8, 11])
def test_uniform_tables(K, R):
    S, J = 5, 777
    off = np.arange(S * J + 1, dtype=np.int64) * K
    for grid in (1, 7, 152):
        p = esp.plan_stream(off, S, J, R, grid, uniform_k=K)
        check(p, off, S, J, None, None, K)
        assert len(p["cta_begin"]) - 1 == min(grid, len(p["tiles"]))


@pytest.mark.parametrize("kmax", [3, 40, 128, 200, 256])
def test_sorted_layout_tables(kmax):
    rng = np.random.default_rng(kmax)
    S, J = 4, 900
    K = rng.integers(1, kmax + 1, size=S * J)
    off0 = np.zeros(S * J + 1, np.int64)
    off0[1:] = np.cumsum(K)
    off, jmap, scen, runk = esp.sort_layout_k(off0, S, J, 256)
    assert np.all(runk > 0)
    for grid in (3, 152):
        p = esp.plan_stream(off, S, J, 6, grid, scen=scen, runk=runk)
        check(p, off, S, J, scen, runk, 0)


def test_heavy_tail_shape():
    t = W.heavy_tail(scenarios=[2, 9], J=6000).table
    off, jmap, scen, runk = esp.sort_layout_k(t.job_off, t.S, t.J, 256)
    p = esp.plan_stream(off, t.S, t.J, t.R, 152, scen=scen, runk=runk)
    check(p, off, t.S, t.J, scen, runk, 0)
    # the per-CTA split is balanced: the largest range's bytes within 5% of the mean
    opt = p["tiles"][:, 4].astype(np.int64)
    per = np.array([opt[p["cta_begin"][c]:p["cta_begin"][c + 1]].sum() for c in range(len(p["cta_begin"]) - 1)])
    assert per.max() <= 1.05 * per.mean() + 2 * p["stage_opt"]


def test_ineligible_tables_are_refused():
    # a job of 300 options is outside every run of the streaming pass
    S, J = 1, 10
    K = np.full(S * J, 5)
    K[4] = 300
    off0 = np.zeros(S * J + 1, np.int64)
    off0[1:] = np.cumsum(K)
    off, jmap, scen, runk = esp.sort_layout_k(off0, S, J, 256)
    assert runk[np.where(jmap == 4)[0][0]] == 0
    with pytest.raises(esp.EspError):
        esp.plan_stream(off, S, J, 6, 10, scen=scen, runk=runk)
    # a uniform K that is not a run size (4 or more options, not a multiple of 4), and one above 256
    for K in (10, 260):
        with pytest.raises(esp.EspError):
            esp.plan_stream(np.arange(11, dtype=np.int64) * K, 1, 10, 6, 4, uniform_k=K)
    # K = 12 is a run size (three groups of four options, four lanes per job)
    p = esp.plan_stream(np.arange(11, dtype=np.int64) * 12, 1, 10, 6, 4, uniform_k=12)
    check(p, np.arange(11, dtype=np.int64) * 12, 1, 10, None, None, 12)


def test_sort_layout_k_default_and_256():
    rng = np.random.default_rng(4)
    S, J = 3, 500
    K = rng.integers(1, 300, size=S * J)
    off0 = np.zeros(S * J + 1, np.int64)
    off0[1:] = np.cumsum(K)
    a = esp.sort_layout(off0, S, J)            # the library's layout: runs of up to 128 options
    b = esp.sort_layout_k(off0, S, J, 128)
    for x, y in zip(a, b):
        assert np.array_equal(x, y)
    # with 256 (the streaming pass's runs): jobs of 129..256 options join padded runs, larger ones keep
    # their size and no run
    off, jmap, scen, runk = esp.sort_layout_k(off0, S, J, 256)
    Kj = K[jmap]
    big = Kj > 256
    assert np.all(runk[big] == 0) and np.all(np.diff(off)[big] == Kj[big])
    mid = (Kj >= 3) & (Kj <= 256)
    assert np.all(runk[mid] == 4 * ((Kj[mid] + 3) // 4)) and np.all(np.diff(off)[mid] == runk[mid])
