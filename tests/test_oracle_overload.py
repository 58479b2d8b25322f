"""The qualitative behaviour the paper states for the price update (Sec. 3.2.3, after Eq. price_update;
the pricing case study of Sec. 5): when GPU memory is over-subscribed its price rises, which moves jobs
to configurations with a smaller memory footprint until the aggregate demand fits; a resource that is
not over-subscribed keeps a zero price. Checked on the oracle (CPU) with a burst of four training jobs
on a two-GPU node, each with a peak configuration and a lower-memory one worth 8-12% less (the
figures of the case study's trade-off; the footprints are ours).

With two options per job and only the memory price moving, the best response has a closed form: job j
leaves its peak configuration exactly when the memory price exceeds its switch price
(v_peak - v_low) / (m_peak - m_low) (Eq. esp_score with the GPU price at 0), so the order and the
rounds of the switches follow from the price trajectory alone."""

import numpy as np

import oracle
from tests.test_oracle_pins import table_from_jobs

GPU_SHARE = 500                         # milli-GPU per job: two jobs share each GPU
JOBS = {                                # name: (peak value, peak GB, lower-memory value, GB)
    "resnet50": (1.00, 24, 0.88, 14),   # AMP
    "bert": (1.00, 36, 0.90, 24),       # activation checkpointing
    "ppo": (1.00, 16, 0.92, 10),        # smaller batch
    "ncf": (1.00, 12, 0.89, 8),         # smaller batch
}
CAPACITY = (2000, 58)                   # two GPUs; 58 GB fits only if every job steps down


def instance():
    jobs = [[(vp, (GPU_SHARE, mp)), (vl, (GPU_SHARE, ml))] for vp, mp, vl, ml in JOBS.values()]
    return table_from_jobs(jobs, CAPACITY)


def switch_prices():
    return np.array([(vp - vl) / (mp - ml) for vp, mp, vl, ml in JOBS.values()])


def test_memory_price_rises_and_steers_jobs_to_lower_memory_until_feasible():
    t = instance()
    T = 300
    sol = oracle.solve_scenario(t, 0, 1e-4, T, mode=oracle.RAW, traces=True, sel_trace=True)
    lam, dem, sel = sol.lambda_trace, sol.demand_trace, sol.sel_trace
    peak_mem = sum(mp for _, mp, _, _ in JOBS.values())
    # at zero prices every job runs its peak configuration, and memory is over-subscribed
    assert np.all(sel[0] == 0) and dem[0, 1] == peak_mem > CAPACITY[1]
    # the GPU share is never over-subscribed, so its price stays 0
    assert np.all(dem[:, 0] == GPU_SHARE * len(JOBS)) and np.all(lam[:, 0] == 0.0)
    # feasibility is reached, and only with every job on its lower-memory configuration
    first = int(np.argmax(dem[:, 1] <= CAPACITY[1]))
    assert dem[first, 1] <= CAPACITY[1] and np.all(sel[first] == 1)
    assert first > 0
    for r in range(first):
        # while memory is over-subscribed its price rises every round ...
        assert lam[r + 1, 1] > lam[r, 1]
        # ... and jobs only ever step down, never back up
        assert np.all(sel[r + 1] >= sel[r])
    # each job steps down in the round its switch price is first exceeded (closed form)
    p = switch_prices()
    for r in range(first + 1):
        assert np.array_equal(sel[r], (lam[r, 1] > p).astype(np.int32)), r
    # the cheapest memory to give up goes first: BERT, ResNet-50, PPO, NCF
    order = [int(np.argmax(sel[:first + 1, j] == 1)) for j in range(len(JOBS))]
    assert np.argsort(order, kind="stable").tolist() == np.argsort(p, kind="stable").tolist()
    assert len(set(order)) == len(JOBS)


def test_no_overload_no_price():
    """With memory for every peak configuration the prices stay 0 and nobody steps down."""
    jobs = [[(vp, (GPU_SHARE, mp)), (vl, (GPU_SHARE, ml))] for vp, mp, vl, ml in JOBS.values()]
    t = table_from_jobs(jobs, (2000, 88))
    sol = oracle.solve_scenario(t, 0, 1e-4, 50, mode=oracle.RAW, traces=True, sel_trace=True)
    assert np.all(sol.lambda_trace == 0.0) and np.all(sol.sel_trace == 0)
    assert sol.feasible == 1
