"""The seeded generators: shapes, determinism, the scenario-subset property and the stated
distributions of the synthetic workloads."""

import numpy as np
import pytest

from paper_2608_07971_gb300 import workloads as W


def test_splitmix64_reference_values():
    # SplitMix64 seeded with 0: first outputs as published with the generator's reference code
    # (state += 0x9E3779B97F4A7C15, then the two xor-shift-multiply rounds).
    def ref(n):
        out, state = [], 0
        for _ in range(n):
            state = (state + 0x9E3779B97F4A7C15) & ((1 << 64) - 1)
            z = state
            z = ((z ^ (z >> 30)) * 0xBF58476D1CE4E5B9) & ((1 << 64) - 1)
            z = ((z ^ (z >> 27)) * 0x94D049BB133111EB) & ((1 << 64) - 1)
            out.append(z ^ (z >> 31))
        return out
    assert ref(1)[0] == 0xE220A8397B1DCDAF
    # draw_bits(seed, stream, n) is output n of a stream whose start state is mix(seed*GAMMA ^ stream)
    start = int(W._mix(np.array([0], np.uint64))[0])  # seed 0, stream 0 -> mix(0) = 0
    assert start == 0
    got = [int(W.draw_bits(0, np.array([0], np.uint64), n)[0]) for n in range(4)]
    assert got == ref(4)


@pytest.mark.parametrize("name,shape", [
    ("tiny_cluster", (1, 64, 4, 4, 512)),
    ("cluster_512", (1, 2048, 6, 6, 32768)),
    ("placement_expanded", (1, 4096, 8, 134, 4096 * 768)),
])
def test_shapes(name, shape):
    t = W.make(name).table
    assert (t.S, t.J, t.R, t.P, t.n_opt) == shape
    assert t.units.dtype == np.int32 and t.units.shape == (t.n_opt, t.R)
    assert t.values.dtype == np.float64 and np.all(np.isfinite(t.values))
    assert np.all(t.units >= 0)
    assert np.all(np.diff(t.job_off) >= 1)
    assert t.capacity.shape == (t.S, t.P) and np.all(t.capacity > 0)


def test_deterministic_and_scenario_subset_identical():
    a = W.whatif_batch(scenarios=[0, 1, 2, 3, 4, 5], J=256).table
    b = W.whatif_batch(scenarios=[4, 1], J=256).table
    for i, s in enumerate([4, 1]):
        sa, sb = a.scenario(s), b.scenario(i)
        assert np.array_equal(sa.units, sb.units)
        assert np.array_equal(sa.values, sb.values)
        assert np.array_equal(sa.job_off, sb.job_off)
        assert np.array_equal(sa.capacity, sb.capacity)
    c = W.whatif_batch(scenarios=[0, 1, 2, 3, 4, 5], J=256).table
    assert np.array_equal(a.units, c.units) and np.array_equal(a.values, c.values)


def test_config_distributions():
    t = W.cluster_512().table
    g = t.units[:, 0]
    assert set(np.unique(g).tolist()) == {1000 * k for k in range(1, 9)}
    assert t.units[:, 1].min() >= 1 and t.units[:, 1].max() <= 163840
    assert t.units[:, 4].max() <= 900 and t.units[:, 5].max() <= 400
    # log-normal(0, 1) base values: the median of b_j is about 1
    b_max = np.array([t.values[t.job_off[j]:t.job_off[j + 1]].max() for j in range(t.J)])
    assert 0.6 < np.median(b_max) < 1.4


def test_whatif_capacity_jitter():
    t = W.whatif_batch(scenarios=range(64), J=64).table
    ratio = t.capacity / np.asarray(W.CAP_512)[None, :]
    assert ratio.min() >= 0.79 and ratio.max() <= 1.21
    assert ratio.std() > 0.05


def test_heavy_tail_counts():
    t = W.heavy_tail(scenarios=[3], J=65536).table
    K = t.option_counts()
    assert K.min() >= 1 and K.max() == 256
    assert abs((K == 256).mean() - 0.1607) < 0.01      # clipped Zipf(1.3) tail mass
    assert abs(K.mean() - 58.5) < 1.5
    # capacity is 60 % of the summed lower-median demand: the argmax-value demand exceeds it
    assert t.capacity.shape == (1, 6)


def test_placement_structure():
    t = W.placement_expanded().table
    n = 768
    assert np.all(t.group[:n] == np.tile(np.arange(64), 12))
    assert np.array_equal(t.units[:n, 6], t.units[:n, 0]) and np.array_equal(t.units[:n, 7], t.units[:n, 1])
    # the interference penalty is in [0, 1) and varies by node
    assert t.r_global == 6 and t.P == 134


def test_iac_rows_ranges_and_job_level_fields():
    J, K = 300, 16
    f = W.iac_rows(6, J, K).astype(np.float64)
    assert f.shape == (J * K, 14) and np.all(np.isfinite(f))
    sm, occ, dram, fb, tc, typ = f[:, 0], f[:, 1], f[:, 2], f[:, 3], f[:, 4], f[:, 5]
    assert np.all((sm >= 0.1) & (sm <= 1.0)) and np.all((occ > 0) & (occ <= sm))
    assert np.all((dram >= 0.05) & (dram <= 0.9)) and np.all((tc >= 0) & (tc <= 0.9))
    assert np.all((fb >= 2048) & (fb <= 78000))
    rows = f.reshape(J, K, 14)
    # type, parameter count, micro-batch, mixed precision, ISL and OSL are per job
    for c in (5, 6, 8, 10, 11, 12):
        assert np.all(rows[:, :, c] == rows[:, :1, c]), c
    train = rows[:, 0, 5] == 0
    assert 0.3 < train.mean() < 0.7
    assert np.all(rows[train][:, :, 11:14] == 0) and np.all(rows[~train][:, :, 8:11] == 0)
    assert np.array_equal(W.iac_rows(6, J, K), W.iac_rows(6, J, K))


def test_iac_pairs_partners_and_scenario_subset():
    S, J, K = 4, 50, 8
    p = W.iac_pairs(6, S, J, K).reshape(S, J, K, 2)
    assert np.all(p[..., 0] == (np.arange(J)[:, None] * K + np.arange(K)[None, :])[None])
    partner_job, partner_cfg = p[..., 1] // K, p[..., 1] % K
    assert np.all(partner_job != np.arange(J)[None, :, None])           # never the job itself
    assert np.all(partner_job == partner_job[..., :1]) and np.all(partner_cfg == partner_cfg[..., :1])
    assert np.all((p >= 0) & (p < J * K))
    # the first scenarios of a larger batch are the smaller batch
    assert np.array_equal(W.iac_pairs(6, 2, J, K), W.iac_pairs(6, S, J, K)[: 2 * J * K])


def test_iac_model_shapes_and_scaling():
    m = W.iac_model(6, 48)
    assert m.W1.shape == (48, 36) and m.W2.shape == (48, 48) and m.W3.shape == (48,)
    assert m.bn1.shape == (4, 48) and m.bn2.shape == (4, 48)
    assert np.all(m.bn1[3] > 0) and np.all(m.bn2[3] > 0)       # running variances
    for a in (m.W1, m.b1, m.bn1, m.W2, m.b2, m.bn2, m.W3):
        assert a.dtype == np.float32 and np.all(np.isfinite(a))
    # the first layer sees inputs of order one: W1 scaled by the inputs' spread
    z = (W.IAC_INPUT_MEAN[None, :] + W.IAC_INPUT_STD[None, :]) @ m.W1.T.astype(np.float64) + m.b1
    assert np.all(np.abs(z) < 20.0)


def test_table_digest_identifies_the_table():
    a = W.whatif_batch(scenarios=[0, 3], J=64).table
    b = W.whatif_batch(scenarios=[0, 3], J=64).table
    assert a.digest() == b.digest() and len(a.digest()) == 64
    # a scenario drawn alone is the same table as that scenario cut from a batch
    assert W.whatif_batch(scenarios=[3], J=64).table.digest() == a.scenario(1).digest()
    units = a.units.copy()
    units[5, 2] += 1
    assert W.OptionTable(**{**a.__dict__, "units": units}).digest() != a.digest()
    values = a.values.copy()
    values[7] = np.nextafter(values[7], np.inf)
    assert W.OptionTable(**{**a.__dict__, "values": values}).digest() != a.digest()
    g = W.placement_expanded(scenarios=[0], J=8).table
    assert g.group is not None and g.digest() != W.OptionTable(**{**g.__dict__, "group": g.group[::-1].copy()}).digest()
