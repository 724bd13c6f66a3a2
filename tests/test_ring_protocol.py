"""Randomized model of the decode kernel's shared-memory ring protocol (host logic only).

The fused decode kernel (paper_2403_06082_gb300/csrc/fq_decode.cu) moves each K block of a task
through a ring of S stages guarded by mbarriers.  A parity wait on an mbarrier is only exact when
the barrier has completed either exactly the phases before the awaited one or one more: a waiter
that is ahead returns at once, and one that has been lapped waits for a later phase.  This test
runs the kernel's roles as coroutines under random delays and asserts, at every wait, that the
barrier is at the awaited phase or one past it; it also checks that every round's MMAs run once
and that the run ends.

Roles and barriers (one round = one K block in one stage):
    weight producer   waits empty[s]; loads the T tile onto fullA[s] or the code block onto cfull[s]
    act. producer     waits empty[s]; loads the activation tile onto fullB[s]
    decoder d         owns stages s = d (mod 4); waits cfull[s] in core rounds, arrives fullA[s]
                      (with decoder pairs two warps own each stage, each expanding half of its
                      rows: fullA then takes two arrivals, and the weight producer adds a plain
                      arrival to its tile's in weight rounds)
    issuer q          owns stages s = q (mod NI); waits fullA[s], fullB[s]; commits empty[s]
"""
import random

import pytest


class Bar:
    def __init__(self, count, name):
        self.count, self.pending, self.done, self.name = count, 0, 0, name

    def arrive(self):
        self.pending += 1
        if self.pending == self.count:
            self.pending = 0
            self.done += 1


def wait(bar, phase, who):
    """Wait for the completion of phase `phase` (0-based) of `bar`, checking exactness."""
    while True:
        d = bar.done
        assert d >= phase, f"{who} ahead of {bar.name}: {d} phases done, waits for {phase}"
        assert d <= phase + 1, f"{who} lapped on {bar.name}: {d} phases done, waits for {phase}"
        if d == phase + 1:
            return
        yield


def run(seed, S, NI, follow_every_round=False, pairs=False):
    rnd = random.Random(seed)
    tasks = [(p, rnd.randint(0, 12)) for p in (0, 1, 2) for _ in range(rnd.randint(0, 4))]
    rounds = [p for p, n in tasks for _ in range(n)]
    full_a = [Bar(2 if pairs else 1, f"fullA{s}") for s in range(S)]
    full_b = [Bar(1, f"fullB{s}") for s in range(S)]
    empty = [Bar(1, f"empty{s}") for s in range(S)]
    cfull = [Bar(1, f"cfull{s}") for s in range(S)]
    landing = []            # [cycles left, barrier] of copies and MMAs in flight
    mma = []

    def delay():
        for _ in range(rnd.randint(0, 4)):
            yield

    def weight_producer():
        for r, p in enumerate(rounds):
            s = r % S
            if r >= S:
                yield from wait(empty[s], r // S - 1, "weight producer")
            yield from delay()
            landing.append([rnd.randint(1, 20), cfull[s] if p == 1 else full_a[s]])
            if pairs and p != 1:
                full_a[s].arrive()          # the producer's second arrival of a weight round

    def act_producer():
        for r, _ in enumerate(rounds):
            s = r % S
            if r >= S:
                yield from wait(empty[s], r // S - 1, "activation producer")
            yield from delay()
            landing.append([rnd.randint(1, 20), full_b[s]])

    def decoder(d, half=0):
        seen = [0] * S
        for r, p in enumerate(rounds):
            s = r % S
            if follow_every_round:
                # the earlier rule: every decoder follows every round's stage release
                if r >= S:
                    yield from wait(empty[s], r // S - 1, f"decoder {d}")
                if s % 4 != d or p != 1:
                    continue
            elif s % 4 != d or p != 1:
                continue
            yield from wait(cfull[s], seen[s], f"decoder {d}.{half}")
            seen[s] += 1
            yield from delay()
            full_a[s].arrive()

    def issuer(q):
        for r, _ in enumerate(rounds):
            s = r % S
            if s % NI != q:
                continue
            yield from wait(full_a[s], r // S, f"issuer {q}")
            yield from wait(full_b[s], r // S, f"issuer {q}")
            yield from delay()
            mma.append(r)
            landing.append([rnd.randint(1, 10), empty[s]])

    alive = [weight_producer(), act_producer()] + [decoder(d) for d in range(4)] + \
            [issuer(q) for q in range(NI)]
    if pairs:
        alive += [decoder(d, 1) for d in range(4)]
    steps = 0
    while alive:
        steps += 1
        assert steps < 100000, f"no progress (seed {seed})"
        for e in list(landing):
            e[0] -= 1
            if e[0] <= 0:
                landing.remove(e)
                e[1].arrive()
        rnd.shuffle(alive)
        for co in list(alive):
            if rnd.random() < 0.3:
                continue
            try:
                next(co)
            except StopIteration:
                alive.remove(co)
    assert sorted(mma) == list(range(len(rounds)))


# ring depths the kernel builds: 8 stages with four issuers (16 and 32 tokens), 5 with one (64)
@pytest.mark.parametrize("S,NI", [(8, 4), (12, 4), (4, 4), (5, 1), (8, 1)])
def test_stage_owned_ring_is_exact(S, NI):
    for seed in range(150):
        run(seed, S, NI)


# four issuers with 16 or 32 tokens run two decoder warps per stage
@pytest.mark.parametrize("S", [12, 8, 4])
def test_stage_owned_ring_with_decoder_pairs_is_exact(S):
    for seed in range(150):
        run(seed, S, 4, pairs=True)


def test_following_every_round_can_be_lapped():
    """The model catches the hazard the stage-owned protocol removes."""
    with pytest.raises(AssertionError, match="lapped|ahead|no progress"):
        for seed in range(300):
            run(seed, 8, 4, follow_every_round=True)
