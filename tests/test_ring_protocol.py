"""Model of the verify kernels' shared-memory ring, on the CPU.

One producer fills slot j % NST with tile j after the slot's previous use was
freed; consumer warp j % CW takes tile j.  Barriers are modelled as the
hardware's phase-parity test: a wait for parity x passes once the completed
phase count P has (P & 1) != x.  Copies complete in random order and warps
run in random order.  The protocol the kernels use (a consumer first waits
for the slot's previous use to be freed, then for its copy) must never let a
warp read a slot that does not hold its tile; the parity-only wait the ring
had before must be caught by the model.
"""
import random

import pytest


class Bar:
    def __init__(self):
        self.phases = 0

    def passed(self, parity):
        return (self.phases & 1) != parity


def run(nst, cw, n_tiles, seed, wait_previous_use):
    rng = random.Random(seed)
    full = [Bar() for _ in range(nst)]
    empty = [Bar() for _ in range(nst)]
    slot_tile = [None] * nst          # the tile whose copy landed in the slot
    in_flight = []                    # (slot, tile) copies issued, not landed
    next_issue = 0
    warp_next = list(range(cw))       # next tile of each warp
    done = 0
    for _ in range(200000):
        if done == n_tiles:
            return True
        moves = []
        j = next_issue
        if j < n_tiles and (j < nst or empty[j % nst].passed(((j // nst) - 1) & 1)):
            moves.append("issue")
        if in_flight:
            moves.append("land")
        for w in range(cw):
            j = warp_next[w]
            if j >= n_tiles:
                continue
            s, use = j % nst, j // nst
            ready = full[s].passed(use & 1)
            if wait_previous_use and use > 0:
                ready = ready and empty[s].passed((use - 1) & 1)
            if ready:
                moves.append(("read", w))
        if not moves:
            return False              # no move possible: the ring stalls
        m = rng.choice(moves)
        if m == "issue":
            in_flight.append((next_issue % nst, next_issue))
            next_issue += 1
        elif m == "land":
            s, tile = in_flight.pop(rng.randrange(len(in_flight)))
            slot_tile[s] = tile
            full[s].phases += 1
        else:
            w = m[1]
            j = warp_next[w]
            s = j % nst
            if slot_tile[s] != j:
                raise AssertionError(f"warp {w} read slot {s} holding tile {slot_tile[s]} for tile {j}")
            empty[s].phases += 1      # the slot is freed
            warp_next[w] += cw
            done += 1
    raise AssertionError("schedule did not finish")


@pytest.mark.parametrize("nst,cw", [(12, 8), (8, 8), (16, 8), (4, 2)])
def test_ring_never_reads_a_wrong_tile(nst, cw):
    for seed in range(300):
        assert run(nst, cw, 200, seed, wait_previous_use=True)


def test_parity_only_wait_is_caught():
    caught = 0
    for seed in range(300):
        try:
            run(12, 8, 200, seed, wait_previous_use=False)
        except AssertionError:
            caught += 1
    assert caught > 0


def test_too_few_slots_for_the_warps_is_caught():
    """6 slots for 8 warps (2 x slots not a multiple of the warps, which the
    kernels' static assert rejects): the previous-use wait is no longer exact."""
    caught = 0
    for seed in range(100):
        try:
            run(6, 8, 200, seed, wait_previous_use=True)
        except AssertionError:
            caught += 1
    assert caught > 0
