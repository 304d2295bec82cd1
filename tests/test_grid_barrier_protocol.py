"""Model of the grid barrier (grid_sync) used by the fused layer tail, on the
CPU: each block reads the generation word, arrives on the counter; the last
arrival resets the counter and advances the generation; the others wait for
the generation to change.  Steps of different blocks interleave at random over
several uses.  No block may leave use k before every block has arrived at use
k, and no schedule may stall.  Reading the generation after arriving instead
can miss the release, which the model must catch as a stall.
"""
import random


def run(n_blocks, uses, seed, read_gen_first=True):
    rng = random.Random(seed)
    count, gen = 0, 0
    # per block: (use, stage, saved gen); stage 0 = before read/arrive, 1 = after
    # first action, 2 = arrived and waiting, 3 = passed
    state = [[0, 0, None] for _ in range(n_blocks)]
    arrived = [0] * uses
    for _ in range(100000):
        live = [b for b in range(n_blocks) if state[b][0] < uses]
        if not live:
            return True
        moves = []
        for b in live:
            use, stage, g = state[b]
            if stage in (0, 1):
                moves.append(b)
            elif stage == 2 and gen != g:
                moves.append(b)
        if not moves:
            return False                                  # every block waits: a stall
        b = rng.choice(moves)
        use, stage, g = state[b]
        if stage == 0:
            if read_gen_first:
                state[b] = [use, 1, gen]                  # read the generation
            else:
                arrived[use] += 1                         # arrive first ...
                count += 1
                if count == n_blocks:
                    count = 0
                    gen += 1
                    state[b] = [use + 1, 0, None]
                else:
                    state[b] = [use, 1, None]
        elif stage == 1:
            if read_gen_first:
                arrived[use] += 1                         # ... then arrive
                count += 1
                if count == n_blocks:                     # the last block releases
                    count = 0
                    gen = g + 1
                    state[b] = [use + 1, 0, None]
                else:
                    state[b] = [use, 2, g]
            else:
                state[b] = [use, 2, gen]                  # reads the generation late
        else:
            assert arrived[use] == n_blocks, "a block left before every block arrived"
            state[b] = [use + 1, 0, None]
    raise AssertionError("schedule did not finish")


def test_grid_barrier_releases_only_complete_uses():
    for seed in range(500):
        assert run(5, 6, seed)


def test_reading_the_generation_late_can_stall():
    assert any(not run(5, 6, seed, read_gen_first=False) for seed in range(500))


def run_after_timeout(n_blocks, uses, seed, stop_and_reset=True):
    """A call in which one block is too slow: at its first barrier the others
    run out of their bounded wait.  With stop_and_reset (the kernels' rule) the
    blocks that timed out leave the kernel, the slow block arrives late, and the
    next call's first kernel zeroes the two words before the barrier is used
    again; otherwise the timed-out blocks carry on into the next use and nothing
    resets.  Then a clean call runs `uses` uses under random interleaving.
    Returns True when every use of the clean call released only after all its
    blocks arrived."""
    rng = random.Random(seed)
    word = {"count": 0, "gen": 0}

    def arrive():   # atomicAdd; the block that reads n - 1 resets the count and releases
        old = word["count"]
        word["count"] = old + 1
        if old == n_blocks - 1:
            word["count"] = 0
            word["gen"] += 1

    # call 1: blocks 1.. arrive at use 0 and time out (the slow block 0 has not arrived)
    for _ in range(1, n_blocks):
        arrive()
    if not stop_and_reset:
        for _ in range(1, n_blocks):             # they go on and arrive at use 1 of call 1
            arrive()
    arrive()                                     # the slow block arrives late
    if stop_and_reset:
        word["count"], word["gen"] = 0, 0        # the next call's first kernel
    count, gen = word["count"], word["gen"]
    # call 2: a clean call from whatever state call 1 left
    arrived = [0] * uses
    state = [[0, 0, None] for _ in range(n_blocks)]
    for _ in range(100000):
        live = [b for b in range(n_blocks) if state[b][0] < uses]
        if not live:
            return True
        moves = [b for b in live if state[b][1] in (0, 1) or (state[b][1] == 2 and gen != state[b][2])]
        if not moves:
            return False
        b = rng.choice(moves)
        use, stage, g = state[b]
        if stage == 0:
            state[b] = [use, 1, gen]
        elif stage == 1:
            arrived[use] += 1
            count += 1
            if count == n_blocks:
                count = 0
                gen = g + 1
                state[b] = [use + 1, 0, None]
            else:
                state[b] = [use, 2, g]
        else:
            if arrived[use] != n_blocks:
                return False                     # released before every block arrived
            state[b] = [use + 1, 0, None]
    raise AssertionError("schedule did not finish")


def test_timed_out_use_then_clean_call():
    for seed in range(300):
        assert run_after_timeout(5, 4, seed)


def test_carrying_on_after_a_timeout_releases_early():
    assert any(not run_after_timeout(5, 4, seed, stop_and_reset=False) for seed in range(300))
