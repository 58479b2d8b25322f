"""The round exchange of the cluster-resident solve (k_resident in csrc/esp_resident.cu), modelled on
the host (no GPU): two buffers of partials, one cluster barrier per round, and every CTA reads its
round's partials exactly, under any interleaving of the CTAs.

Per round r each CTA of a cluster of C stores its partial (demand columns, and the hash and dual
when traced) into slot [r mod 2][its rank] of every CTA's shared memory, all CTAs meet at the
cluster barrier, and each then sums the C slots [r mod 2][0 .. C-1] of its own shared memory in rank
order and applies the price update. Two buffers suffice because a CTA stores into buffer r mod 2
again only in round r + 2, after the barrier of round r + 1, which every CTA reaches only after it
finished reading round r's slots. A stopped scenario skips its work but not its barriers (the stop
is decided from identical totals in every CTA). The model steps the CTAs in a random order (memory
sequentially consistent; the barrier's release and acquire order it in the kernel) and checks every
read; the one-buffer control must fail."""

import numpy as np
import pytest


def simulate(rng, C, T, n_buf=2, stop_at=None):
    """True if every CTA read every round's partials exactly."""
    part = rng.integers(0, 1 << 40, size=(T, C))
    buf = np.zeros((C, n_buf, C), np.int64)      # buf[reader][parity][writer]
    arrived = 0
    state = [[0, 0] for _ in range(C)]           # round, step (0 store, 1 arrive, 2 wait, 3 read)
    ok = True
    while True:
        live = [c for c in range(C) if state[c][0] < T]
        if not live:
            return ok
        movable = [c for c in live if not (state[c][1] == 2 and arrived < (state[c][0] + 1) * C)]
        assert movable, "the barrier cannot deadlock: every CTA meets it once per round"
        c = movable[rng.integers(len(movable))]
        r, step = state[c]
        working = stop_at is None or r < stop_at
        if step == 0 and working:
            for reader in range(C):
                buf[reader, r % n_buf, c] = part[r, c]
        elif step == 1:
            arrived += 1
        elif step == 3 and working:
            ok &= bool(np.array_equal(buf[c, r % n_buf], part[r]))
        state[c] = [r + 1, 0] if step == 3 else [r, step + 1]


@pytest.mark.parametrize("C", [1, 2, 4, 8, 16])
def test_two_buffers_carry_every_round(C):
    rng = np.random.default_rng(C)
    for _ in range(30):
        assert simulate(rng, C, T=10)
    assert simulate(rng, C, T=10, stop_at=4)   # stopped rounds: barriers only


def test_one_buffer_races():
    """The control: with one buffer a CTA that runs ahead overwrites a slot a slower CTA has not read."""
    rng = np.random.default_rng(3)
    assert not all(simulate(rng, 4, T=8, n_buf=1) for _ in range(100))
