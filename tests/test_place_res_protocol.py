"""The round protocol of the grid-resident placement solve (k_place_res in csrc/esp_place.cu), modelled
on the host (no GPU): its rotation of demand buffers gives every CTA exactly its round's totals,
under any interleaving of the CTAs.

Per round r every CTA adds its jobs' demand to buffer r mod 3 (atomics), arrives at the grid barrier
and waits until all G CTAs have arrived r + 1 times, then reads the totals of buffer r mod 3 for the
price update; after that barrier CTA 0 also clears buffer (r + 2) mod 3, the one of round r - 1,
whose last reads happened before each CTA arrived at barrier r. A CTA may run ahead into round r + 1
(adding to buffer (r + 1) mod 3) while slower CTAs still read round r's totals, which is why a third
buffer is needed: with two, CTA 0's clearing of round r - 1's buffer would meet the fast CTAs' adds
of round r + 1. The model steps the CTAs in a random order, one action at a time (memory is
sequentially consistent here; the kernel orders it with a fence before each arrival and an acquire
load in the wait), and checks every read against the round's true totals; the two-buffer control
must fail."""

import numpy as np
import pytest


def simulate(rng, G, T, n_buf=3):
    """Runs the protocol; returns True if every CTA read every round's exact totals."""
    contrib = rng.integers(0, 1000, size=(T, G))
    buf = np.zeros(n_buf, np.int64)
    bar = 0
    # per CTA: round, step (0 add, 1 arrive, 2 wait, 3 read, 4 clear, then the next round)
    state = [[0, 0] for _ in range(G)]
    ok = True
    while True:
        live = [c for c in range(G) if state[c][0] < T]
        if not live:
            return ok
        movable = []
        for c in live:
            r, step = state[c]
            if step == 2 and bar < (r + 1) * G:
                continue                          # waits at the barrier
            movable.append(c)
        assert movable, "every CTA waits: the barrier cannot deadlock when all arrive"
        c = movable[rng.integers(len(movable))]
        r, step = state[c]
        if step == 0:
            buf[r % n_buf] += contrib[r, c]
        elif step == 1:
            bar += 1
        elif step == 3:
            ok &= bool(buf[r % n_buf] == contrib[r].sum())
        elif step == 4 and c == 0:
            buf[(r + n_buf - 1) % n_buf] = 0      # round r - 1's buffer ((r + 2) mod 3 for three)
        state[c] = [r + 1, 0] if step == 4 else [r, step + 1]


@pytest.mark.parametrize("G", [1, 2, 3, 19, 152])
def test_three_buffers_give_every_round_its_totals(G):
    rng = np.random.default_rng(G)
    for _ in range(20 if G < 100 else 3):
        assert simulate(rng, G, T=12)


def test_two_buffers_race():
    """The control: with two buffers some interleaving lets a fast CTA's adds for round r + 1 land in
    the buffer CTA 0 is about to clear (or read stale totals)."""
    rng = np.random.default_rng(5)
    assert not all(simulate(rng, 4, T=8, n_buf=2) for _ in range(200))
