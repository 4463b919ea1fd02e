"""Per-layer expert cache oracle: LRU / LFU / FIFO replacement, fetch accounting and metrics.

Section 4.1 "Simulation": each layer keeps B routed experts (K <= B < E); caches start empty and
persist; first fills count as misses; each miss is one expert fetch plus, when the cache is full, an
eviction under LRU, LFU or FIFO; the hit rate and fetches per token follow Eq. metrics (f = K - h at
batch size 1).

The paper only runs batch size 1 with K distinct experts per step. The rule used for any batch, per
layer and decode step t (it reduces to the paper's at batch 1):

1. U = the distinct experts chosen by any token of the step; each expert of U counts one access.
2. Every expert of U already cached is a hit and gets last_use = t.
3. The other experts of U are misses, taken in ascending expert id. Each is one fetch. It goes to
   the lowest-numbered free slot if there is one; otherwise it replaces, among slots with
   last_use < t (not used at this step), the one with the smallest policy key:
     LRU:  (last_use, expert id)
     LFU:  (accesses of the expert since the stream began, last_use, expert id)
     FIFO: (step the expert was inserted, expert id)
   If every slot was used at step t (only possible when |U| > B) the expert is fetched for this
   step only ("bypass") and not cached.
4. h = |U and cache|, f = |U| - h.

Readings: LFU counts persist across evictions (the paper evicts "the least frequently accessed
experts"); FIFO hits do not refresh the insertion order; ties always fall to the older use and
then the lower expert id.

Prefetch (offloading systems load experts ahead of need, Section 2; the paper gives no rule): a
prefetch is a cache event of its own between two steps, with its own time stamp, given a ranked
list of candidate experts (the predicted ones, most likely first) and a cap n_max <= B on loads.
Every candidate already cached is touched (last use = the event; no access is counted, so LFU
counts stay those of real steps), so no load of this event evicts it. The first n_max candidates
not cached are loaded, in ascending id: each takes the lowest free slot or evicts, among slots not
touched at this event, the smallest policy key (an insertion stamps last use and insertion with
the event); if no slot qualifies the expert is skipped. Each load is one prefetch fetch. A
prefetched expert that the next step uses is a hit of that step and counts as a useful prefetch.
Prefetched experts the next step does not use are dropped when it begins (their slots become
free before its hits and misses are processed), so a wrong prediction can be cancelled while its
bytes are still in flight; the pending set is cleared at every step.

Two independent formulations are given: ``SlotCache`` (per-slot arrays and an argmin of the policy
key) and ``OrderedCache`` (an ordered list of cached experts kept in victim order). Tests require
them to agree.
"""
from __future__ import annotations

import numpy as np


POLICIES = ("LRU", "LFU", "FIFO")


class SlotCache:
    """B slots as tag / last-use / insertion arrays plus per-expert access counts; the victim is the
    argmin of the policy key over slots not used at this step."""

    def __init__(self, E: int, B: int, policy: str = "LRU"):
        if not (0 < B < E):
            raise ValueError("need 0 < B < E")
        if policy not in POLICIES:
            raise ValueError(f"unknown policy {policy}")
        self.E, self.B, self.policy = E, B, policy
        self.tag = [-1] * B
        self.last = [-1] * B
        self.ins = [-1] * B
        self.freq = [0] * E
        self.t = 0
        self.pf = set()      # experts loaded by prefetch since the last step (still cached)
        self.prefetched = 0  # prefetch loads so far
        self.useful = 0      # prefetched experts used by the step that followed

    def _key(self, s):
        e = self.tag[s]
        if self.policy == "LRU":
            return (self.last[s], e)
        if self.policy == "LFU":
            return (self.freq[e], self.last[s], e)
        return (self.ins[s], e)

    def step(self, ids):
        """Process one decode step given every expert id chosen by its tokens.

        Returns (hits, fetches, bypass, misses) where misses lists (expert, slot) in processing
        order, slot = -1 for a bypass fetch.
        """
        t = self.t
        U = sorted(set(int(e) for e in np.asarray(ids).reshape(-1)))
        for e in U:
            if not 0 <= e < self.E:
                raise ValueError(f"expert id {e} out of range")
        for e in U:
            self.freq[e] += 1
        self.useful += len(self.pf & set(U))
        for s in range(self.B):  # unused prefetched experts are dropped
            if self.tag[s] in self.pf and self.tag[s] not in U:
                self.tag[s], self.last[s], self.ins[s] = -1, -1, -1
        self.pf = set()
        hits = 0
        for s in range(self.B):
            if self.tag[s] in U:
                self.last[s] = t
                hits += 1
        misses = []
        for e in U:
            if e in self.tag:
                continue
            slot = self._claim(t)
            if slot is None:
                misses.append((e, -1))
                continue
            self._insert(slot, e, t)
            misses.append((e, slot))
        self.t += 1
        bypass = sum(1 for _, s in misses if s < 0)
        return hits, len(misses), bypass, misses

    def _claim(self, t):
        """Slot for an insertion at event t: the lowest free slot, else the smallest policy key
        among slots not touched at t, else None."""
        free = [s for s in range(self.B) if self.tag[s] < 0]
        if free:
            return free[0]
        cand = [s for s in range(self.B) if self.last[s] < t]
        return min(cand, key=self._key) if cand else None

    def _insert(self, slot, e, t):
        self.pf.discard(self.tag[slot])
        self.tag[slot] = e
        self.last[slot] = t
        self.ins[slot] = t

    def prefetch(self, candidates, n_max=None):
        """Prefetch event for the ranked candidate list (distinct ids, most likely first), loading
        at most n_max (default B) of them. Returns the (expert, slot) loads in processing order."""
        t = self.t
        cand = _check_candidates(candidates, self.E)
        n_max = self.B if n_max is None else n_max
        if not 1 <= n_max <= self.B:
            raise ValueError("a prefetch loads between 1 and B experts")
        for s in range(self.B):
            if self.tag[s] in cand:
                self.last[s] = t
        P = sorted([e for e in cand if e not in self.tag][:n_max])
        loads = []
        for e in P:
            slot = self._claim(t)
            if slot is None:
                continue
            self._insert(slot, e, t)
            self.pf.add(e)
            loads.append((e, slot))
        self.t += 1
        self.prefetched += len(loads)
        return loads


def _check_candidates(candidates, E):
    cand = [int(e) for e in candidates]
    if len(set(cand)) != len(cand) or any(not 0 <= e < E for e in cand):
        raise ValueError("prefetch candidates must be distinct valid expert ids")
    return cand


class LRUStamps(SlotCache):
    """SlotCache with LRU replacement."""

    def __init__(self, E: int, B: int):
        super().__init__(E, B, "LRU")


class OrderedCache:
    """Cached experts kept in a list ordered by eviction preference (first = next victim).

    LRU: touched experts move to the end; FIFO: only insertions append; LFU: the list is kept
    sorted by (accesses, last use, id) by re-inserting an expert at its place (bisection) whenever
    it is touched. Experts touched in the current step are never victims.
    """

    def __init__(self, E: int, B: int, policy: str = "LRU"):
        if not (0 < B < E):
            raise ValueError("need 0 < B < E")
        if policy not in POLICIES:
            raise ValueError(f"unknown policy {policy}")
        self.E, self.B, self.policy = E, B, policy
        self.order = []          # cached experts, next victim first
        self.keys = []           # LFU only: sort keys parallel to order
        self.slot_of = {}        # expert -> slot
        self.free = list(range(B))
        self.count = [0] * E
        self.t = 0
        self.pf = set()
        self.prefetched = 0
        self.useful = 0

    def _place(self, e):
        """(Re)insert e at its position in the victim order after it was touched at step t."""
        if self.policy == "LFU":
            k = (self.count[e], self.t, e)
            lo, hi = 0, len(self.keys)
            while lo < hi:
                mid = (lo + hi) // 2
                if self.keys[mid] < k:
                    lo = mid + 1
                else:
                    hi = mid
            self.keys.insert(lo, k)
            self.order.insert(lo, e)
        else:
            self.order.append(e)

    def _remove(self, e):
        i = self.order.index(e)
        self.order.pop(i)
        if self.policy == "LFU":
            self.keys.pop(i)

    def step(self, ids):
        U = sorted(set(int(e) for e in np.asarray(ids).reshape(-1)))
        for e in U:
            if not 0 <= e < self.E:
                raise ValueError(f"expert id {e} out of range")
        for e in U:
            self.count[e] += 1
        self.useful += sum(1 for e in U if e in self.pf)
        for e in sorted(self.pf - set(U)):  # unused prefetched experts are dropped
            self._remove(e)
            self.free.append(self.slot_of.pop(e))
        self.free.sort()
        self.pf = set()
        touched = set()
        hits = 0
        for e in U:
            if e in self.slot_of:
                hits += 1
                self._touch(e, touched)
        misses = []
        for e in U:
            if e in self.slot_of:
                continue
            slot = self._take_slot(touched)
            if slot is None:
                misses.append((e, -1))
                continue
            self.slot_of[e] = slot
            touched.add(e)
            self._place(e)
            misses.append((e, slot))
        self._end_event(touched)
        bypass = sum(1 for _, s in misses if s < 0)
        return hits, len(misses), bypass, misses

    def _touch(self, e, touched):
        touched.add(e)
        if self.policy != "FIFO":
            self._remove(e)
            self._place(e)

    def _take_slot(self, touched):
        """A free slot, else the slot of the first expert in victim order not touched at this
        event (evicting it), else None."""
        if self.free:
            return self.free.pop(0)
        victim = next((v for v in self.order if v not in touched), None)
        if victim is None:
            return None
        self._remove(victim)
        self.pf.discard(victim)
        return self.slot_of.pop(victim)

    def _end_event(self, touched):
        if self.policy == "LRU":
            # experts touched at one event: lower id first (older) among equal last use
            tail = [v for v in self.order if v in touched]
            head = [v for v in self.order if v not in touched]
            self.order = head + sorted(tail)
        self.t += 1

    def prefetch(self, candidates, n_max=None):
        """Prefetch event (see the module header); returns the (expert, slot) loads."""
        cand = _check_candidates(candidates, self.E)
        n_max = self.B if n_max is None else n_max
        if not 1 <= n_max <= self.B:
            raise ValueError("a prefetch loads between 1 and B experts")
        touched = set()
        for e in sorted(cand):
            if e in self.slot_of:
                self._touch(e, touched)
        P = sorted([e for e in cand if e not in self.slot_of][:n_max])
        loads = []
        for e in P:
            slot = self._take_slot(touched)
            if slot is None:
                continue
            self.slot_of[e] = slot
            touched.add(e)
            self._place(e)
            self.pf.add(e)
            loads.append((e, slot))
        self._end_event(touched)
        self.prefetched += len(loads)
        return loads

    def state(self):
        """(tag per slot) for comparison with SlotCache."""
        tag = [-1] * self.B
        for e, s in self.slot_of.items():
            tag[s] = e
        return tag


class LRUList(OrderedCache):
    """OrderedCache with LRU replacement."""

    def __init__(self, E: int, B: int):
        super().__init__(E, B, "LRU")


def simulate(steps_ids, E: int, B: int, cls=SlotCache, policy: str = "LRU", prefetch=None):
    """Run one layer's cache over a stream of steps; steps_ids[t] holds the ids chosen at step t
    and, when given, prefetch[t] = (ranked candidates, n_max) of a prefetch just before step t
    (None: no prefetch event).

    Returns per-step arrays hits, fetches, bypass and the list of per-step miss lists.
    """
    c = cls(E, B, policy)
    h, f, b, ml = [], [], [], []
    for t, ids in enumerate(steps_ids):
        if prefetch is not None and prefetch[t] is not None:
            c.prefetch(*prefetch[t])
        hi, fi, bi, mi = c.step(ids)
        h.append(hi)
        f.append(fi)
        b.append(bi)
        ml.append(mi)
    return np.array(h), np.array(f), np.array(b), ml


def metrics(total_hits, total_fetches, N: int, L: int, K: int):
    """Eq. metrics at batch size 1: HR = sum h / (N L K), Fetches/tok = sum f / N."""
    return total_hits / (N * L * K), total_fetches / N


def fetches_per_token_from_hit_rate(hr, L: int, K: int):
    """The identity Fetches/tok = L K (1 - HR) that follows from f = K - h (Eq. metrics)."""
    return L * K * (1.0 - hr)
