"""The stage-ring protocol of the tcgen05 expert GEMM with LoRA adapters (csrc/gemm_tc.cu), modelled
on the CPU: a producer thread fills TMA stages, a builder warp fills each adapted tile's extra
k-block, and the MMA thread consumes every stage in order. Stage barriers are waited on by phase
parity, which identifies a phase only within one phase of the barrier's progress: a waiter two
phases ahead passes at once, two phases behind it never passes. The model checks, over random
interleavings of the three threads, that every wait of the kernel's hand-off design stays within
one phase and that every stage is consumed; and that the two designs the kernel no longer uses
(a builder waiting only for its own stage, a builder waiting on every stage in lockstep) break
the rule, so the check can tell them apart."""
import random

import pytest

STAGES = 4


class Ambiguous(AssertionError):
    pass


def _seq(kblocks, adapted):
    s = []
    for a in adapted:
        s += ["T"] * kblocks + (["L"] if a else [])
    return s


def _run(kblocks, adapted, builder, seed):
    """Random interleaving of producer, builder and MMA; builder is "handoff" (the kernel's),
    "own-stage" or "lockstep". Raises Ambiguous if a parity wait is two phases off."""
    rnd = random.Random(seed)
    seq = _seq(kblocks, adapted)
    n = len(seq)
    done = {("e", s): 0 for s in range(STAGES)}  # completed phases of each barrier
    done.update({("f", s): 0 for s in range(STAGES)})
    done.update({("g", j): 0 for j in range(2)})

    def wait(bar, phase):  # wait for completion of `phase` (0-based)
        d = done[bar]
        if not phase - 1 <= d <= phase + 1:
            raise Ambiguous((bar, phase, d))
        return d >= phase + 1

    lstages = [i for i, k in enumerate(seq) if k == "L"]
    prod = mma = 0
    nl_p = nl_b = 0  # hand-offs made / taken
    build = 0        # stage index of the lockstep / own-stage builders
    for _ in range(10 ** 6):
        if mma == n:
            return True
        c = rnd.randrange(3)
        if c == 0 and prod < n:  # producer: waits each stage's empty phase (round r waits r - 1)
            r, s = divmod(prod, STAGES)
            if seq[prod] == "L" and builder != "handoff":
                prod += 1  # the other designs let the builder take that stage alone
                continue
            if r == 0 or wait(("e", s), r - 1):
                if seq[prod] == "T":
                    done[("f", s)] += 1
                else:
                    done[("g", nl_p & 1)] += 1
                    nl_p += 1
                prod += 1
        elif c == 1:
            if builder == "handoff" and nl_b < len(lstages):
                if wait(("g", nl_b & 1), nl_b >> 1):
                    done[("f", lstages[nl_b] % STAGES)] += 1
                    nl_b += 1
            elif builder == "lockstep" and build < n:
                r, s = divmod(build, STAGES)
                if r == 0 or wait(("e", s), r - 1):
                    if seq[build] == "L":
                        done[("f", s)] += 1
                    build += 1
            elif builder == "own-stage" and nl_b < len(lstages):
                it = lstages[nl_b]
                r, s = divmod(it, STAGES)
                if r == 0 or wait(("e", s), r - 1):
                    done[("f", s)] += 1
                    nl_b += 1
        elif c == 2:  # MMA: waits each stage's full phase in order, then frees it
            r, s = divmod(mma, STAGES)
            if wait(("f", s), r):
                done[("e", s)] += 1
                mma += 1
    raise AssertionError("no progress")


PATTERNS = [[1] * 6, [1, 0, 1, 1, 0, 0, 1], [0, 1], [1], [1, 1, 0, 1]]


@pytest.mark.parametrize("kblocks", [2, 3, 4, 8, 22, 64])
def test_handoff_waits_stay_within_one_phase(kblocks):
    for adapted in PATTERNS:
        for seed in range(20):
            assert _run(kblocks, adapted, "handoff", seed)


@pytest.mark.parametrize("builder", ["own-stage", "lockstep"])
def test_earlier_builders_break_the_rule(builder):
    """Tiles of 64 k-blocks (Mixtral GEMM13): both earlier designs make an ambiguous wait."""
    broken = 0
    for seed in range(20):
        try:
            _run(64, [1, 1, 1], builder, seed)
        except Ambiguous:
            broken += 1
    assert broken == 20
