"""Host-side checks of the C-ABI library that need no GPU: it loads, exports every function that
include/*.h declares, reports no GPU cleanly, and its tile planner covers every job exactly once."""

import ctypes
import os
import re

import numpy as np
import pytest

from paper_2608_07971_gb300 import esp, workloads as W

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    from paper_2608_07971_gb300 import build
    build.build()
    return esp.load_library()


def declared_functions():
    names = []
    for h in ("esp.h", "esp_debug.h", "esp_iac.h"):
        src = open(os.path.join(ROOT, "include", h)).read()
        src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
        names += re.findall(r"^\s*(?:const\s+)?\w+\s*\*?\s*(esp_\w+)\s*\(", src, flags=re.M)
    return sorted(set(names))


def test_exports_every_declared_function(lib):
    names = declared_functions()
    assert len(names) >= 15
    for n in names:
        assert hasattr(lib, n), n
    assert set(names) == set(esp.EXPORTED)


def test_status_strings(lib):
    for s in range(9):
        assert esp.esp_status_string(s)
    assert esp.esp_status_string(99) == "unknown status"


def test_create_without_gpu_is_unsupported(lib):
    import torch
    if torch.cuda.is_available():
        pytest.skip("a GPU is present")
    h = ctypes.c_void_p()
    assert lib.esp_create(ctypes.byref(h), -1, None) == esp.ESP_ERR_UNSUPPORTED
    assert lib.esp_create(None, -1, None) == esp.ESP_ERR_INVALID_ARG


def test_null_context_rejected(lib):
    assert lib.esp_solve(None, None, None) == esp.ESP_ERR_INVALID_ARG
    assert lib.esp_get_prices(None, None) == esp.ESP_ERR_INVALID_ARG
    assert lib.esp_debug_set_pdl(None, 1) == esp.ESP_ERR_INVALID_ARG
    assert lib.esp_debug_set_plan_waves(None, 2) == esp.ESP_ERR_INVALID_ARG
    assert lib.esp_load_placement(None, 1, 1, 1, 1, 2, 1, None, None, None, None, 1, None, None, None) \
        == esp.ESP_ERR_INVALID_ARG
    lib.esp_destroy(None)


def test_null_predictor_rejected(lib):
    assert lib.esp_iac_create(None, -1, None) == esp.ESP_ERR_INVALID_ARG
    assert lib.esp_iac_set_path(None, 0) == esp.ESP_ERR_INVALID_ARG
    assert lib.esp_iac_synchronize(None) == esp.ESP_ERR_INVALID_ARG
    assert lib.esp_iac_load_model(None, 8, None, None, None, None, None, None, None, 0.0, 1e-5) \
        == esp.ESP_ERR_INVALID_ARG
    assert lib.esp_iac_predict(None, 0, None, 0, None, 1.0, None) == esp.ESP_ERR_INVALID_ARG
    assert lib.esp_iac_predict_host(None, 0, None, 0, None, 1.0, None) == esp.ESP_ERR_INVALID_ARG
    n = ctypes.c_int64(5)
    assert lib.esp_iac_last_launch_count(None, ctypes.byref(n)) == esp.ESP_ERR_INVALID_ARG
    lib.esp_iac_destroy(None)


def test_create_predictor_without_gpu_is_unsupported(lib):
    import torch
    if torch.cuda.is_available():
        pytest.skip("a GPU is present")
    h = ctypes.c_void_p()
    assert lib.esp_iac_create(ctypes.byref(h), -1, None) == esp.ESP_ERR_UNSUPPORTED
    assert h.value is None


def tiles_cover(job_off, S, J, tiles, wb, tile_opt):
    """Independent re-check of a plan: each job once, in order, chunks contiguous and complete."""
    opt_begin = tiles[:, 0].astype(np.int64) & 0xFFFFFFFF | (tiles[:, 1].astype(np.int64) << 32)
    job_begin = tiles[:, 2].astype(np.int64) & 0xFFFFFFFF | (tiles[:, 3].astype(np.int64) << 32)
    n_opt, n_job, scen, flags = tiles[:, 4], tiles[:, 5], tiles[:, 6], tiles[:, 7]
    covered = np.zeros(S * J, np.int64)  # options covered per job
    for k in range(len(tiles)):
        assert 1 <= n_opt[k] <= tile_opt
        if flags[k] & 1:  # big chunk
            j = job_begin[k]
            covered[j] += n_opt[k]
            assert job_off[j] <= opt_begin[k] and opt_begin[k] + n_opt[k] <= job_off[j + 1]
        else:
            j0, j1 = job_begin[k], job_begin[k] + n_job[k]
            assert opt_begin[k] == job_off[j0] and opt_begin[k] + n_opt[k] == job_off[j1]
            covered[j0:j1] += np.diff(job_off[j0:j1 + 1])
            assert np.all(np.arange(j0, j1) // J == scen[k])
    assert np.array_equal(covered, np.diff(job_off))
    assert wb[0] == 0 and wb[-1] == len(tiles) and np.all(np.diff(wb) >= 0)


@pytest.mark.parametrize("case", ["uniform16", "zipf", "big", "mixed", "ones"])
def test_planner_covers_every_job(lib, case):
    rng = np.random.default_rng(5)
    S, J = 3, 500
    if case == "uniform16":
        K = np.full(S * J, 16)
    elif case == "zipf":
        K = np.minimum(256, rng.zipf(1.3, S * J))
    elif case == "big":
        K = rng.choice([1, 700, 768, 1500], S * J)
    elif case == "mixed":
        K = rng.integers(1, 300, S * J)
    else:
        K = np.ones(S * J, np.int64)
    off = np.zeros(S * J + 1, np.int64)
    off[1:] = np.cumsum(K)
    for tile_opt in (32, 256):
        for warps in (1, 7, 64, 5000):
            tiles, wb = esp.plan(off, S, J, tile_opt, warps)
            assert len(wb) - 1 <= warps
            tiles_cover(off, S, J, tiles, wb, tile_opt)


def tile_cost(tiles):
    """The planner's cost estimate, restated: 1050 + 1650 per row (+850 for the last chunk of a large
    job); a row is 128 options (chunks, runs of 4m-option jobs: 32 / 2^ceil(log2 m) jobs) or 32."""
    fl, n_opt, n_job = tiles[:, 7], tiles[:, 4].astype(np.int64), tiles[:, 5].astype(np.int64)
    big, run = (fl & 1) != 0, (fl & 8) != 0
    k = (fl >> 8) & 255
    lanes = np.array([1 << int(np.ceil(np.log2(max(1, kk // 4)))) if kk >= 4 else 1 for kk in k])
    rows = np.where(big, (n_opt + 127) // 128,
                    np.where(run & (k >= 4), (n_job + 32 // lanes - 1) // (32 // lanes), (n_opt + 31) // 32))
    return 1050 + 1650 * rows + np.where((fl & 4) != 0, 850, 0)


def test_planner_balances_cost(lib):
    """Warp ranges have about equal estimated cost: the spread is at most a few tiles' cost, every
    option is covered, and no range starts inside the chunks of a large job."""
    t = W.whatif_batch(scenarios=range(16), J=2048).table
    for tile_opt, warps in ((256, 600), (128, 3000)):
        tiles, wb = esp.plan(t.job_off, t.S, t.J, tile_opt, warps)
        cost = tile_cost(tiles)
        per_warp = np.array([cost[wb[w]:wb[w + 1]].sum() for w in range(len(wb) - 1)])
        assert tiles[:, 4].sum() == t.n_opt
        assert per_warp.max() - per_warp.min() <= cost.max()
    rng = np.random.default_rng(3)
    S, J = 4, 3000
    K = np.minimum(256, rng.zipf(1.3, S * J))
    off = np.zeros(K.size + 1, np.int64)
    off[1:] = np.cumsum(K)
    soff, jmap, scen, runk = esp.sort_layout(off, S, J)
    tiles, wb = esp.plan_runs(soff, scen, runk, S, J, 128, 257)
    cost = tile_cost(tiles)
    per_warp = np.array([cost[wb[w]:wb[w + 1]].sum() for w in range(len(wb) - 1)])
    # each boundary sits within about one job of two chunks of its target
    assert per_warp.max() - per_warp.min() <= 4 * cost.max()
    for w in range(1, len(wb) - 1):
        assert not (tiles[wb[w], 7] & 1) or (tiles[wb[w], 7] & 2)


def test_planner_rejects_bad_offsets(lib):
    off = np.array([0, 3, 3, 5], np.int64)   # an empty job
    with pytest.raises(esp.EspError):
        esp.plan(off, 1, 3, 32, 4)


def test_tile_options(lib):
    assert lib.esp_debug_tile_options(6, 0) == 256
    assert lib.esp_debug_tile_options(4, 0) % 32 == 0
    assert lib.esp_debug_tile_options(8, 1) % 32 == 0


def expected_sorted_order(K, S, J):
    """The sorted layout's job order, restated: per scenario the 3..128-option jobs by padded size
    (4 * ceil(K / 4)), stable; then per scenario the larger jobs; then per scenario the 2-option and
    the 1-option jobs."""
    order, padded, runk = [], [], []
    for s in range(S):
        js = range(s * J, (s + 1) * J)
        small = sorted((j for j in js if 3 <= K[j] <= 128), key=lambda j: (-(-K[j] // 4), j))
        for j in small:
            order.append(j); padded.append(4 * -(-K[j] // 4)); runk.append(4 * -(-K[j] // 4))
    for s in range(S):
        for j in range(s * J, (s + 1) * J):
            if K[j] > 128:
                order.append(j); padded.append(K[j]); runk.append(0)
    for s in range(S):
        for k in (2, 1):
            for j in range(s * J, (s + 1) * J):
                if K[j] == k:
                    order.append(j); padded.append(k); runk.append(k)
    return np.array(order), np.array(padded), np.array(runk)


@pytest.mark.parametrize("case", ["zipf", "mixed", "small", "big"])
def test_sorted_layout(lib, case):
    rng = np.random.default_rng(11)
    S, J = 3, 400
    if case == "zipf":
        K = np.minimum(256, rng.zipf(1.3, S * J))
    elif case == "mixed":
        K = rng.integers(1, 300, S * J)
    elif case == "small":
        K = rng.integers(1, 6, S * J)
    else:
        K = rng.choice([129, 255, 700, 3], S * J)
    off = np.zeros(S * J + 1, np.int64)
    off[1:] = np.cumsum(K)
    soff, jmap, scen, runk = esp.sort_layout(off, S, J)
    order, padded, want_runk = expected_sorted_order(K, S, J)
    assert np.array_equal(jmap, order)                       # a permutation in the stated order
    assert np.array_equal(np.diff(soff), padded)             # padding to a multiple of 4 (3..128)
    assert np.array_equal(runk, want_runk)
    assert np.array_equal(scen, order // J)
    part_a = runk >= 4
    assert np.all(soff[:-1][part_a] % 4 == 0)               # every padded job starts 4-aligned
    assert np.all(np.diff(soff) >= K[jmap])
    for tile_opt in (128,):
        for warps in (1, 9, 200):
            tiles, wb = esp.plan_runs(soff, scen, runk, S, J, tile_opt, warps)
            opt_begin = tiles[:, 0].astype(np.int64) & 0xFFFFFFFF | (tiles[:, 1].astype(np.int64) << 32)
            job_begin = tiles[:, 2].astype(np.int64) & 0xFFFFFFFF | (tiles[:, 3].astype(np.int64) << 32)
            covered = np.zeros(S * J, np.int64)
            for k in range(len(tiles)):
                fl = tiles[k, 7]
                if fl & 1:
                    covered[job_begin[k]] += tiles[k, 4]
                    continue
                j0, j1 = job_begin[k], job_begin[k] + tiles[k, 5]
                covered[j0:j1] += np.diff(soff[j0:j1 + 1])
                assert np.all(scen[j0:j1] == tiles[k, 6])
                if fl & 8:                                   # a run tile: one option count
                    kk = (fl >> 8) & 0xFFF
                    assert np.all(runk[j0:j1] == kk) and tiles[k, 4] == kk * (j1 - j0)
                    if kk >= 4:
                        assert opt_begin[k] % 4 == 0
                else:
                    assert np.all(runk[j0:j1] == 0)
            assert np.array_equal(covered, np.diff(soff))


def test_host_formulas_match_the_oracle(lib):
    """esp_adaptive_threshold and esp_effective_capacity (host code of the library) give the oracle's
    values bit for bit."""
    import oracle
    rng = np.random.default_rng(21)
    tb = rng.random(50) + 1.0
    for util, beta_max in ((0.93, 0.05), (0.4, 0.2), (1.7, 0.1)):
        got = esp.esp_adaptive_threshold(tb, 0.3, util, 0.8, beta_max)
        want = np.array([oracle.adaptive_threshold(x, 0.3, util, 0.8, beta_max) for x in tb])
        assert np.array_equal(got, want)
    K = rng.integers(1, 5, 40)
    q_off = np.zeros(41, np.int64)
    q_off[1:] = np.cumsum(K)
    q_units = rng.integers(0, 1000, (int(q_off[-1]), 6)).astype(np.int32)
    cap = rng.integers(10000, 40000, 6).astype(np.int64)
    for gamma in (0.0, 0.37, 1.0):
        assert np.array_equal(esp.esp_effective_capacity(cap, q_off, q_units, gamma),
                              oracle.effective_capacity(cap, q_off, q_units, gamma))
    with pytest.raises(esp.EspError):
        esp.esp_effective_capacity(cap, np.array([0, 0], np.int64), q_units, 0.5)   # an empty queued job
    # capacities must be exact in fp64 (the floor then stays inside int64) and positive
    edge = cap.copy()
    edge[2] = 1 << 53
    assert np.array_equal(esp.esp_effective_capacity(edge, q_off, q_units, 0.0), edge)
    for bad in (0, -5, (1 << 53) + 1, np.iinfo(np.int64).max):
        edge[2] = bad
        with pytest.raises(esp.EspError):
            esp.esp_effective_capacity(edge, q_off, q_units, 0.5)
