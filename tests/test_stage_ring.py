"""Host model of the C-Block kernel's stage ring: TMA-issuing producers, one MMA consumer, and the
per-stage `full` / `empty` mbarriers waited on by phase parity.

A parity wait on an mbarrier passes when the barrier's current (incomplete) phase has the other
parity, so a waiter two phases ahead of the barrier sees "complete".  The kernel gives every stage one
producer thread (stage s is filled by producer s % n, n dividing the stage count), so each thread
waits on its stages in order and is never more than one phase ahead.  The model runs random
interleavings of the producers and the consumer and checks that the consumer always reads the k-block
it expects.  It also shows what that rule avoids: k-blocks dealt round-robin (it % n) stay safe only
while n is at most the stage count (each producer's previous k-block gates its next wait), and break
with more producers than stages -- 4 producers on the 3-stage ring of the 256-column tiles, the
configuration that failed on the GPU.
"""
import random

import pytest


class Barrier:
    def __init__(self):
        self.phase = 0  # completed phases; every barrier here has an arrival count of 1

    def try_wait_parity(self, parity):
        return (self.phase & 1) != parity

    def arrive(self):
        self.phase += 1


def run_ring(stages, producers, n_kb, owner, seed):
    """Random interleaving; returns the first (k-block, value read) mismatch, or None."""
    rng = random.Random(seed)
    full = [Barrier() for _ in range(stages)]
    empty = [Barrier() for _ in range(stages)]
    slot = [None] * stages
    todo = {p: [it for it in range(n_kb) if owner(it) == p] for p in range(producers)}
    consumed = 0
    steps = 0
    while consumed < n_kb:
        steps += 1
        if steps > 200 * n_kb:
            return consumed, "stuck"  # no actor can pass its wait any more
        actors = [p for p in range(producers) if todo[p]] + ["mma"]
        a = rng.choice(actors)
        if a == "mma":
            it = consumed
            s = it % stages
            if full[s].try_wait_parity((it // stages) & 1):
                if slot[s] != it:
                    return it, slot[s]
                consumed += 1
                empty[s].arrive()
        else:
            it = todo[a][0]
            s = it % stages
            if empty[s].try_wait_parity(((it // stages) & 1) ^ 1):
                slot[s] = it
                full[s].arrive()
                todo[a].pop(0)
    return None


def producers_for(stages):
    """The kernel's producer count for a ring of `stages` stages (tc_producers): one per stage up to
    four stages (the 256-column tiles' four, the packed-weight ring's three), else two."""
    return stages if stages <= 4 else 2


@pytest.mark.parametrize("stages", [3, 4, 6])
def test_stage_owned_by_one_producer_is_safe(stages):
    n = producers_for(stages)
    assert stages % n == 0 and n <= 4
    for seed in range(300):
        assert run_ring(stages, n, 40, lambda it: (it % stages) % n, seed) is None


def test_single_producer_is_safe():
    for seed in range(100):
        assert run_ring(6, 1, 40, lambda it: 0, seed) is None


def test_round_robin_with_at_most_as_many_producers_as_stages_is_safe():
    for stages, n in ((3, 2), (3, 3), (4, 4), (6, 4), (6, 6)):
        for seed in range(150):
            assert run_ring(stages, n, 40, lambda it: it % n, seed) is None, (stages, n, seed)


def test_round_robin_with_more_producers_than_stages_fails():
    for stages, n in ((3, 4), (2, 3), (6, 7)):
        bad = [run_ring(stages, n, 40, lambda it: it % n, seed) for seed in range(150)]
        assert any(b is not None for b in bad), (stages, n)
