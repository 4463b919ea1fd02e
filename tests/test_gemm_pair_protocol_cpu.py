"""The barrier protocol of the CTA-pair expert GEMM (gemm_tc_pair_kernel in csrc/gemm_tc.cu),
modelled on the CPU: two producers (one per CTA of the cluster) load every stage, with both CTAs'
bytes counted on the leader's full[s]; the leader's MMA thread consumes the stages in order and
its commits arrive on empty[s] and tfull[b] of both CTAs; each CTA's four epilogue warps release
an accumulator on the leader's tempty[b] (eight arrivals). Copies land and commits complete at
random later times. Over random interleavings the model checks that nothing deadlocks, that
every parity wait is within one phase of its barrier (a parity identifies a phase only that far),
and that every arrival and every landed byte count goes to the phase it belongs to: in
particular that a CTA's copy for a stage's next round can never land on the leader's barrier
before the round it would corrupt has completed."""
import random

import pytest


class ProtocolError(AssertionError):
    pass


def _run(tiles, kblocks, stages, seed, peer_waits_empty=True):
    rnd = random.Random(seed)
    n = tiles * kblocks  # stage iterations per producer
    done = {}  # completed phases of each barrier

    def bar(name):
        return done.setdefault(name, 0)

    def waited(name, phase):  # wait for completion of `phase` (0-based), by parity
        d = bar(name)
        if not phase - 1 <= d <= phase + 1:
            raise ProtocolError(f"parity wait on {name} for phase {phase} with {d} completed")
        return d >= phase + 1

    # full[s] (leader): one arrival (the leader's expect) and two landings per phase
    pending_full = {}

    def full_event(s, phase, what):
        if bar(("full", s)) != phase:
            raise ProtocolError(f"{what} of round {phase} on full[{s}] during phase {bar(('full', s))}")
        got = pending_full.setdefault(s, set())
        if what in got:
            raise ProtocolError(f"{what} twice in one phase of full[{s}]")
        got.add(what)
        if got == {"arrive", "land0", "land1"}:
            done[("full", s)] += 1
            pending_full[s] = set()

    tempty_count = {0: 0, 1: 0}

    def tempty_arrive(b, phase):
        if bar(("tempty", b)) != phase:
            raise ProtocolError(f"tempty[{b}] arrival for phase {phase} during {bar(('tempty', b))}")
        tempty_count[b] += 1
        if tempty_count[b] == 8:
            tempty_count[b] = 0
            done[("tempty", b)] += 1

    events = []  # (kind, args): copies landing, commits completing
    prod = [0, 0]
    mma_it, mma_tile, mma_k = 0, 0, 0
    mma_waiting_tempty = True
    epi = {(r, w): 0 for r in (0, 1) for w in range(4)}  # tiles finished per epilogue warp

    for _ in range(10 ** 6):
        if all(p == n for p in prod) and mma_tile == tiles and not events and \
                all(v == tiles for v in epi.values()):
            return True
        moves = []
        for r in (0, 1):  # producers
            it = prod[r]
            if it < n:
                s, rd = it % stages, it // stages
                if rd == 0 or (r == 1 and not peer_waits_empty) or waited(("empty", r, s), rd - 1):
                    moves.append(("prod", r))
        if mma_tile < tiles:  # the leader's MMA thread
            b = mma_tile % 2
            if mma_waiting_tempty:
                if mma_tile < 2 or waited(("tempty", b), mma_tile // 2 - 1):
                    moves.append(("mma_acc",))
            else:
                s, rd = mma_it % stages, mma_it // stages
                if waited(("full", s), rd):
                    moves.append(("mma_k",))
        for (r, w), t in epi.items():  # epilogue warps
            if t < tiles and waited(("tfull", r, t % 2), t // 2):
                moves.append(("epi", r, w))
        if events:
            moves.append(("event",))
        if not moves:
            raise ProtocolError("deadlock")
        m = rnd.choice(moves)
        if m[0] == "prod":
            r = m[1]
            it = prod[r]
            s, rd = it % stages, it // stages
            if r == 0:
                full_event(s, rd, "arrive")
            events.append(("land", r, s, rd))
            prod[r] += 1
        elif m[0] == "mma_acc":
            mma_waiting_tempty = False
        elif m[0] == "mma_k":
            s, rd = mma_it % stages, mma_it // stages
            events.append(("commit_empty", s, rd))
            mma_it += 1
            mma_k += 1
            if mma_k == kblocks:
                events.append(("commit_tfull", mma_tile % 2, mma_tile // 2))
                mma_k = 0
                mma_tile += 1
                mma_waiting_tempty = True
        elif m[0] == "epi":
            r, w = m[1], m[2]
            t = epi[(r, w)]
            tempty_arrive(t % 2, t // 2)  # local (leader) or remote (peer) arrival
            epi[(r, w)] += 1
        else:
            ev = events.pop(rnd.randrange(len(events)))
            if ev[0] == "land":
                _, r, s, rd = ev
                full_event(s, rd, f"land{r}")
            elif ev[0] == "commit_empty":  # multicast: both CTAs' empty[s]
                _, s, rd = ev
                for r in (0, 1):
                    if bar(("empty", r, s)) != rd:
                        raise ProtocolError(f"empty[{s}] of CTA {r} out of order")
                    done[("empty", r, s)] += 1
            else:  # commit_tfull, multicast
                _, b, rd = ev
                for r in (0, 1):
                    if bar(("tfull", r, b)) != rd:
                        raise ProtocolError(f"tfull[{b}] of CTA {r} out of order")
                    done[("tfull", r, b)] += 1
    raise ProtocolError("no progress bound reached")


@pytest.mark.parametrize("tiles,kblocks,stages", [(1, 1, 6), (3, 2, 6), (5, 22, 6), (7, 3, 4),
                                                  (2, 64, 6), (9, 1, 2)])
def test_pair_protocol_random_interleavings(tiles, kblocks, stages):
    for seed in range(40):
        assert _run(tiles, kblocks, stages, seed)


def test_model_catches_a_peer_that_skips_its_empty_wait():
    """The check is not vacuous: a peer producer that reuses a stage without waiting for the
    leader's MMAs to free it lets its copy for the next round land on the leader's full[s] while
    the current round is still filling, which the model reports."""
    caught = 0
    for seed in range(40):
        try:
            _run(4, 3, 2, seed, peer_waits_empty=False)
        except ProtocolError:
            caught += 1
    assert caught > 0
