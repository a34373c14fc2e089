"""Host model of the deterministic backward schedule (no GPU).

The cluster backward's deterministic mode (lmhead_bwd4.cu) hands each of its C
clusters (a multiple of 4) quad slot c % 4 of every group of four 512-token
quads and the vocab blocks m, m + C/4, ... (m = c / 4), walked group by group
and, inside a group, block by block.  For every unit a cluster drains one slab
per 256-column job of H into dhidden (the unit's quad) and then one into dW
(the unit's vocab block); a drain waits until the slab's turn counter equals
its position (the block index for dhidden, the quad index for dW) and raises it
by one afterwards.

This model runs those event sequences under random interleavings and checks
that (1) every cluster finishes (no wait-for cycle), and (2) every slab receives
its contributions in the intended order: dhidden in vocab-block order, dW in
token-quad order, whatever the cluster count.  It restates the schedule, not
the kernel: the GPU tests check that the kernel's results do not depend on the
cluster count, bit for bit.
"""
import random

import pytest


def units(c, n_clusters, n_quads, n_blocks):
    """The units (quad, block) of cluster c, in its order."""
    slot, m, n_classes = c % 4, c // 4, n_clusters // 4
    for g in range((n_quads + 3) // 4):
        q = 4 * g + slot
        if q < n_quads:
            for b in range(m, n_blocks, n_classes):
                yield q, b


def simulate(n_clusters, n_quads, n_blocks, n_jobs, seed, schedule=units):
    events = []
    for c in range(n_clusters):
        seq = []
        for q, b in schedule(c, n_clusters, n_quads, n_blocks):
            seq += [("dh", q, j, b) for j in range(n_jobs)]
            seq += [("dw", b, j, q) for j in range(n_jobs)]
        events.append(seq)
    rnd = random.Random(seed)
    pos = [0] * n_clusters
    turn, order = {}, {}
    left = sum(len(s) for s in events)
    while left:
        progressed = False
        for c in rnd.sample(range(n_clusters), n_clusters):
            for _ in range(rnd.randint(1, 3)):
                if pos[c] == len(events[c]):
                    break
                kind, key, j, p = events[c][pos[c]]
                if turn.get((kind, key, j), 0) != p:
                    break                        # not this drain's turn yet
                turn[(kind, key, j)] = p + 1
                order.setdefault((kind, key, j), []).append(p)
                pos[c] += 1
                left -= 1
                progressed = True
        if not progressed:
            return None                          # every unfinished cluster waits
    return order


@pytest.mark.parametrize("n_clusters", [4, 8, 16, 36])
def test_turns_never_deadlock_and_fix_the_order(n_clusters):
    for n_quads in (1, 2, 3, 5, 7, 23):
        for n_blocks in (1, 2, 9, 10, 19, 40):
            for n_jobs in (1, 3):
                order = simulate(n_clusters, n_quads, n_blocks, n_jobs, seed=n_quads * 100 + n_blocks)
                assert order is not None, (n_clusters, n_quads, n_blocks, n_jobs)
                for (kind, _, _), got in order.items():
                    assert got == list(range(n_blocks if kind == "dh" else n_quads))


def test_every_unit_is_scheduled_once():
    for n_clusters in (4, 8, 36):
        seen = [u for c in range(n_clusters) for u in units(c, n_clusters, 23, 297)]
        assert sorted(seen) == [(q, b) for q in range(23) for b in range(297)]


def test_a_wrong_position_is_caught():
    """The model itself can fail: a drain order that cannot be met (dW in
    reverse quad order) leaves every cluster waiting."""
    def reversed_units(c, n_clusters, n_quads, n_blocks):
        for q, b in units(c, n_clusters, n_quads, n_blocks):
            yield n_quads - 1 - q, b

    for n_quads in (5, 8):
        assert simulate(8, n_quads, 4, 1, seed=1, schedule=reversed_units) is None
