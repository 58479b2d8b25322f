"""The allocation-free best response (esp_evaluate_noalloc) against the oracle and esp_evaluate.

esp_evaluate_noalloc serves callers that cannot allocate device memory at the point of use (another
framework's allocator owns the device, or a loop that must not stall on cudaMalloc): they pass every
buffer, and the library's only scratch is a fixed array in its own device memory. On two calls in a
row (the array keeps the previous call's contents) its selections, demands and minimal reduced costs
must equal, bit for bit, the oracle's best response of every scenario at the same prices (Sec. 3.2.2's
per-job subproblem, ties to the lowest local index) and the context-based esp_evaluate. Also covered:
a batch without jobs, a job without options, and more jobs than the kernel's grid holds warps (the
grid-stride loop). The file is named to be collected last, and it passes alone in a fresh process as
well as after the other tests.
"""

import numpy as np
import pytest

import oracle
from paper_2608_07971_gb300 import esp, workloads as W

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def torch():
    t = pytest.importorskip("torch")
    if not t.cuda.is_available():
        pytest.skip("needs a GPU")
    from paper_2608_07971_gb300 import build
    build.build()
    esp.load_library()
    return t


def tables():
    rng = np.random.default_rng(11)
    yield W.whatif_batch(scenarios=[5, 6, 7], J=512).table              # K = 16, duplicates
    t = W.random_table(rng, S=3, J=400, R=6, kmin=1, kmax=300)          # ragged jobs
    for j in range(0, t.S * t.J, 5):                                    # plus exact duplicates
        a, b = t.job_off[j], t.job_off[j + 1]
        t.units[a + 1:b] = t.units[a]
        t.values[a + 1:b] = t.values[a]
    yield t


def prices(rng, t, mode):
    scale = 50.0 if mode == esp.ESP_PRICE_NORMALIZED else 1e-5
    lam = rng.exponential(scale, size=(t.S, t.P))
    lam[rng.random(lam.shape) < 0.2] = 0.0
    return lam


def noalloc(torch, t, d, lam, mode, with_min=True):
    dev = torch.device("cuda", 0)
    sel = torch.full((t.S, t.J), -7, dtype=torch.int32, device=dev)
    dem = torch.full((t.S, t.P), -7, dtype=torch.int64, device=dev)
    ms = torch.full((t.S, t.J), float("nan"), dtype=torch.float64, device=dev) if with_min else None
    lam_d = torch.from_numpy(np.ascontiguousarray(lam)).to(dev)
    stream = torch.cuda.current_stream(dev)
    esp.esp_evaluate_noalloc(t.S, t.J, t.R, d["off"], d["units"], d["values"], d["cap"], lam_d, mode,
                             sel, dem, ms, stream.cuda_stream)
    stream.synchronize()
    return sel.cpu().numpy(), dem.cpu().numpy(), (ms.cpu().numpy() if with_min else None)


def device_table(torch, t):
    dev = torch.device("cuda", 0)
    return {k: torch.from_numpy(np.ascontiguousarray(a)).to(dev) for k, a in
            dict(off=t.job_off, units=t.units, values=t.values, cap=t.capacity).items()}


def oracle_best(t, lam, mode):
    ot = oracle.OracleTable(t)
    out = [oracle.best_response(ot, s, lam[s], mode=mode) for s in range(t.S)]
    return (np.stack([o[0] for o in out]), np.stack([o[1] for o in out]), np.stack([o[2] for o in out]))


@pytest.mark.parametrize("mode", [esp.ESP_PRICE_NORMALIZED, esp.ESP_PRICE_RAW])
def test_noalloc_equals_oracle_on_two_calls(torch, mode):
    rng = np.random.default_rng(5)
    for t in tables():
        solver = esp.Solver(t, device=0)
        d = device_table(torch, t)
        for call in range(2):
            lam = prices(rng, t, mode)
            sel, dem, ms = noalloc(torch, t, d, lam, mode)
            o_sel, o_dem, o_ms = oracle_best(t, lam, mode)
            assert np.array_equal(sel, o_sel), f"selection differs from the oracle on call {call}"
            assert np.array_equal(dem, o_dem), f"demand differs from the oracle on call {call}"
            assert np.array_equal(ms, o_ms), f"minimal reduced cost differs from the oracle on call {call}"
            ref_sel, ref_dem, ref_ms = solver.evaluate(lam, mode=mode)
            assert np.array_equal(sel, ref_sel) and np.array_equal(dem, ref_dem) and np.array_equal(ms, ref_ms)
        solver.close()


def test_noalloc_grid_stride_and_no_min_score(torch):
    # 2 x 300,000 jobs: more than the 65,536 CTAs x 8 warps of the launch, so warps take several jobs
    rng = np.random.default_rng(8)
    S, J, R = 2, 300_000, 4
    K = rng.integers(1, 4, size=S * J)
    off = np.zeros(S * J + 1, np.int64)
    off[1:] = np.cumsum(K)
    n = int(off[-1])
    t = W.OptionTable(S=S, J=J, R=R, P=R, r_global=R, job_off=off,
                      units=rng.integers(0, 5000, size=(n, R)).astype(np.int32),
                      values=rng.lognormal(0.0, 1.0, size=n), group=None,
                      capacity=np.full((S, R), 10**9, np.int64))
    d = device_table(torch, t)
    for call in range(2):
        lam = prices(rng, t, esp.ESP_PRICE_NORMALIZED)
        sel, dem, _ = noalloc(torch, t, d, lam, esp.ESP_PRICE_NORMALIZED, with_min=False)
        o_sel, o_dem, _ = oracle_best(t, lam, esp.ESP_PRICE_NORMALIZED)
        assert np.array_equal(sel, o_sel), f"selection differs from the oracle on call {call}"
        assert np.array_equal(dem, o_dem), f"demand differs from the oracle on call {call}"


def test_noalloc_empty_batch_and_empty_job(torch):
    dev = torch.device("cuda", 0)
    rng = np.random.default_rng(9)
    # J = 0: no job, the demand is overwritten with zeros
    cap = torch.full((3, 4), 100, dtype=torch.int64, device=dev)
    lam = torch.ones((3, 4), dtype=torch.float64, device=dev)
    dem = torch.full((3, 4), -7, dtype=torch.int64, device=dev)
    off = torch.zeros(1, dtype=torch.int64, device=dev)
    esp.esp_evaluate_noalloc(3, 0, 4, off, None, None, cap, lam, esp.ESP_PRICE_RAW, dem, dem, None, None)
    torch.cuda.synchronize()
    assert np.array_equal(dem.cpu().numpy(), np.zeros((3, 4), np.int64))
    # a job without options among normal ones: it chooses nothing and adds no demand
    t = W.random_table(rng, S=2, J=50, R=4, kmin=1, kmax=9)
    K = np.diff(t.job_off)
    K[[3, 77]] = 0
    off = np.zeros(t.S * t.J + 1, np.int64)
    off[1:] = np.cumsum(K)
    keep = np.ones(len(t.values), bool)
    for j in (3, 77):
        keep[t.job_off[j]:t.job_off[j + 1]] = False
    e = W.OptionTable(S=t.S, J=t.J, R=t.R, P=t.P, r_global=t.r_global, job_off=off, units=t.units[keep],
                      values=t.values[keep], group=None, capacity=t.capacity)
    lam = prices(rng, e, esp.ESP_PRICE_NORMALIZED)
    sel, dem, ms = noalloc(torch, e, device_table(torch, e), lam, esp.ESP_PRICE_NORMALIZED)
    assert sel.ravel()[3] == -1 and sel.ravel()[77] == -1
    assert np.isinf(ms.ravel()[3]) and np.isinf(ms.ravel()[77])
    # every other job equals the oracle's answer on the table without the two empty jobs
    full = np.ones(t.S * t.J, bool)
    full[[3, 77]] = False
    o_sel, o_dem, o_ms = oracle_best(t, lam, esp.ESP_PRICE_NORMALIZED)
    o_dem = o_dem.copy()
    for j in (3, 77):
        s = j // t.J
        o_dem[s] -= t.units[t.job_off[j] + o_sel.ravel()[j]]
    assert np.array_equal(sel.ravel()[full], o_sel.ravel()[full])
    assert np.array_equal(ms.ravel()[full], o_ms.ravel()[full])
    assert np.array_equal(dem, o_dem)


def test_noalloc_rejects_oversized_batches(torch):
    dev = torch.device("cuda", 0)
    S, J, R = 20000, 1, 4          # S*R = 80000 prices > the 65536 the scratch array holds
    x = torch.zeros(8, dtype=torch.int64, device=dev)
    with pytest.raises(esp.EspError) as e:
        esp.esp_evaluate_noalloc(S, J, R, x, x, x, x, x, esp.ESP_PRICE_RAW, x, x, None, None)
    assert e.value.status == esp.ESP_ERR_INVALID_ARG
