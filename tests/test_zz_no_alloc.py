"""The allocation-free best response (esp_evaluate_noalloc) against esp_evaluate.

esp_evaluate_noalloc serves callers that cannot allocate device memory at the point of use (another
framework's allocator owns the device, or a loop that must not stall on cudaMalloc): they pass every
buffer, and the library's only scratch is a fixed array in its own device memory. This checks, on two
calls in a row (the array keeps the previous call's contents), that its selections, demands and
minimal reduced costs equal those of the context-based esp_evaluate. The file is named to be
collected last, and it passes alone in a fresh process as well as after the other tests.
"""

import numpy as np
import pytest

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


@pytest.mark.parametrize("mode", [esp.ESP_PRICE_NORMALIZED, esp.ESP_PRICE_RAW])
def test_noalloc_equals_evaluate_on_two_calls(torch, mode):
    dev = torch.device("cuda", 0)
    rng = np.random.default_rng(5)
    for t in tables():
        solver = esp.Solver(t, device=0)
        d = {k: torch.from_numpy(np.ascontiguousarray(a)).to(dev) for k, a in
             dict(off=t.job_off, units=t.units, values=t.values, cap=t.capacity).items()}
        scale = 50.0 if mode == esp.ESP_PRICE_NORMALIZED else 1e-5
        for call in range(2):
            lam = rng.exponential(scale, size=(t.S, t.P))
            lam[rng.random(lam.shape) < 0.2] = 0.0
            ref_sel, ref_dem, ref_ms = solver.evaluate(lam, mode=mode)
            sel = torch.full((t.S, t.J), -1, dtype=torch.int32, device=dev)
            dem = torch.full((t.S, t.P), -7, dtype=torch.int64, device=dev)
            ms = torch.full((t.S, t.J), float("nan"), dtype=torch.float64, device=dev)
            lam_d = torch.from_numpy(lam).to(dev)
            stream = torch.cuda.current_stream(dev)
            esp.esp_evaluate_noalloc(t.S, t.J, t.R, d["off"], d["units"], d["values"], d["cap"], lam_d, mode,
                                     sel, dem, ms, stream.cuda_stream)
            stream.synchronize()
            assert np.array_equal(sel.cpu().numpy(), ref_sel), f"selection differs on call {call}"
            assert np.array_equal(dem.cpu().numpy(), ref_dem), f"demand differs on call {call}"
            assert np.array_equal(ms.cpu().numpy(), ref_ms), f"minimal reduced cost differs on call {call}"
        solver.close()


def test_noalloc_rejects_oversized_batches(torch):
    dev = torch.device("cuda", 0)
    S, J, R = 20000, 1, 4          # S*R = 80000 prices > the 65536 the scratch array holds
    x = torch.zeros(8, dtype=torch.int64, device=dev)
    with pytest.raises(esp.EspError) as e:
        esp.esp_evaluate_noalloc(S, J, R, x, x, x, x, x, esp.ESP_PRICE_RAW, x, x, None, None)
    assert e.value.status == esp.ESP_ERR_INVALID_ARG
