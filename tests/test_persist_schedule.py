"""The persistent evaluation pass's hand-out and release protocol, modelled on the host (no GPU): it
always completes, under any interleaving of the warps.

The model follows k_pass_persist (csrc/esp_pass.cuh) step by step, with the arithmetic left out:
- work items q = 0, 1, ... are (round q / NR, plan range item_order[q mod NR]) pairs, taken from one
  counter in increasing order; the ranges of a round are ordered by the scenario of their first tile;
  a warp reserves its next index one take ahead (the counter's latency is hidden behind a tile), so it
  always holds one index it has not queued yet;
- a warp keeps up to 8 taken items and, before it evaluates tile v, takes more until it knows v + 3
  tiles (the copy pipeline's lookahead); taking never waits;
- it evaluates its tiles in order; on a tile of another scenario or round it first flushes its arrivals
  (tiles evaluated) for the scenario and round it leaves, then waits until the new scenario's prices
  for that round are released;
- the arrival that completes a scenario's tile count for a round applies the price update and
  releases the next round (ver[s] = r + 1).
Warps advance one step at a time in a random order (any interleaving the hardware could produce). The
model checks that every run ends with every scenario released for every round, that no tile is
evaluated before its scenario's prices for that round exist, and, as a control, that the order the
kernel avoids (waiting for the new scenario before flushing the old one) deadlocks."""

import numpy as np
import pytest

QUEUE = 8       # kPersistQueue
LOOKAHEAD = 3   # a warp at tile v takes items until it knows v + kStages + 1 tiles (kStages = 2)


def make_plan(rng, S, max_tiles, NR, parts=1):
    """Tiles of S scenarios cut into NR contiguous ranges; the ranges of a round ordered by the scenario
    of their first tile (stable). parts = 1: each scenario's tiles contiguous (a uniform table);
    parts = 3: the table in three parts, each holding a share of every scenario's tiles in scenario
    order (a sorted layout: runs, chunked jobs, one- and two-option jobs)."""
    tiles_per = rng.integers(1, max_tiles + 1, S)
    if parts == 1:
        scen = np.repeat(np.arange(S), tiles_per)
    else:
        share = [rng.multinomial(t, np.ones(parts) / parts) for t in tiles_per]
        scen = np.concatenate([np.repeat(np.arange(S), [sh[p] for sh in share]) for p in range(parts)])
    n = len(scen)
    cuts = np.sort(rng.choice(np.arange(1, n), size=min(NR - 1, n - 1), replace=False)) if n > 1 else []
    begin = np.concatenate([[0], cuts, [n]]).astype(int)
    NR = len(begin) - 1
    order = sorted(range(NR), key=lambda i: scen[begin[i]])
    return scen, begin, order, np.bincount(scen, minlength=S)


def simulate(rng, scen, begin, order, scen_tiles, T, W, flush_first=True, max_steps=2_000_000):
    S = len(scen_tiles)
    NR = len(order)
    Q = T * NR
    counter = 0
    arrivals = np.zeros((S, T), int)
    ver = np.zeros(S, int)
    warps = [{"tiles": [], "v": 0, "cur": None, "count": 0, "done": False, "pend": None} for _ in range(W)]

    def reserve():
        nonlocal counter
        counter += 1
        return counter - 1

    for w in warps:                              # each warp's first index, requested at entry
        w["pend"] = reserve()

    def take(w):
        # queue occupancy: the items taken whose tiles are not all evaluated
        while len(w["tiles"]) < w["v"] + LOOKAHEAD and w["pend"] < Q:
            ahead_items = len({it for (_, _, it) in w["tiles"][w["v"]:]})
            if ahead_items >= QUEUE:
                break
            q = w["pend"]
            w["pend"] = reserve()                # the index after it, requested now
            r, i = q // NR, order[q % NR]
            w["tiles"].extend((int(scen[k]), r, q) for k in range(begin[i], begin[i + 1]))

    def flush(w):
        """The warp's arrivals for the scenario and round it leaves; True if any were added."""
        added = w["cur"] is not None and w["count"] > 0
        if added:
            s, r = w["cur"]
            arrivals[s, r] += w["count"]
            assert arrivals[s, r] <= scen_tiles[s]
            if arrivals[s, r] == scen_tiles[s]:
                assert ver[s] == r
                ver[s] = r + 1                   # the last arriver's price update releases round r + 1
        w["count"] = 0
        w["cur"] = None
        return added

    for _ in range(max_steps):
        live = [w for w in warps if not w["done"]]
        if not live:
            break
        progressed = False
        for k in rng.permutation(len(live)):
            w = live[k]
            take(w)
            if w["v"] == len(w["tiles"]):        # nothing left to take or evaluate
                flush(w)
                w["done"] = True
                progressed = True
                break
            s, r, _ = w["tiles"][w["v"]]
            if w["cur"] != (s, r):
                if flush_first and flush(w):     # arrivals added (maybe a release): progress
                    progressed = True
                    break
                if ver[s] < r:                   # wait for the scenario's prices of round r
                    continue
                if not flush_first:
                    flush(w)
                w["cur"] = (s, r)
            assert ver[s] >= r                   # prices of round r exist before its tiles are evaluated
            w["count"] += 1
            w["v"] += 1
            progressed = True
            break
        if not progressed:
            return False, arrivals, ver          # every live warp waits: deadlock
    assert all(w["done"] for w in warps)
    return True, arrivals, ver


@pytest.mark.parametrize("parts", [1, 3])
@pytest.mark.parametrize("seed", range(20))
def test_every_interleaving_completes(seed, parts):
    rng = np.random.default_rng(seed)
    S = int(rng.integers(1, 9))
    scen, begin, order, scen_tiles = make_plan(rng, S, int(rng.integers(1, 40)), int(rng.integers(1, 24)), parts)
    T = int(rng.integers(1, 7))
    W = int(rng.integers(1, 12))
    ok, arrivals, ver = simulate(rng, scen, begin, order, scen_tiles, T, W)
    assert ok, "deadlock"
    assert np.array_equal(arrivals, np.repeat(scen_tiles[:, None], T, axis=1))
    assert np.all(ver == T)


def test_one_scenario_many_warps_and_more_warps_than_ranges():
    rng = np.random.default_rng(99)
    for S, tiles, NR, W in ((1, 64, 16, 40), (3, 5, 20, 64), (16, 30, 8, 3)):
        scen, begin, order, scen_tiles = make_plan(rng, S, tiles, NR)
        for _ in range(3):
            ok, arrivals, ver = simulate(rng, scen, begin, order, scen_tiles, 5, W)
            assert ok and np.all(ver == 5)


def test_waiting_before_the_flush_deadlocks():
    """The control: a warp that waits for its next scenario's prices while still holding arrivals of
    the scenario it leaves can block the release it waits for (the ordering the kernel avoids)."""
    rng = np.random.default_rng(7)
    dead = 0
    for _ in range(40):
        scen, begin, order, scen_tiles = make_plan(rng, 2, 6, 4)
        ok, _, _ = simulate(rng, scen, begin, order, scen_tiles, 4, 2, flush_first=False)
        dead += not ok
    assert dead > 0
