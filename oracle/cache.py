"""Per-layer expert cache oracle: LRU replacement, fetch accounting and metrics.

Section 4.1 "Simulation": each layer keeps B routed experts (K <= B < E); caches start empty and
persist; first fills count as misses; each miss is one expert fetch plus, when the cache is full, an
eviction; the hit rate and fetches per token follow Eq. metrics (f = K - h at batch size 1).

The paper only runs batch size 1 with K distinct experts per step. The rule used for any batch, per
layer and decode step t (it reduces to the paper's at batch 1):

1. U = the distinct experts chosen by any token of the step.
2. Every expert of U already cached is a hit and gets last_use = t.
3. The other experts of U are misses, taken in ascending expert id. Each is one fetch. It goes to
   the lowest-numbered free slot if there is one; otherwise it replaces the slot whose
   (last_use, expert id) is smallest among slots with last_use < t; if every slot was used at step t
   (only possible when |U| > B) the expert is fetched for this step only ("bypass") and not cached.
4. h = |U and cache|, f = |U| - h.

Two independent formulations are given: ``LRUStamps`` (per-slot timestamps and an argmin) and
``LRUList`` (a recency-ordered list). Tests require them to agree.
"""
from __future__ import annotations

import numpy as np


class LRUStamps:
    """LRU cache of B slots as tag/timestamp arrays; victim = argmin (last_use, expert id)."""

    def __init__(self, E: int, B: int):
        if not (0 < B < E):
            raise ValueError("need 0 < B < E")
        self.E, self.B = E, B
        self.tag = [-1] * B
        self.last = [-1] * B
        self.t = 0

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
        hits = 0
        for s in range(self.B):
            if self.tag[s] in U:
                self.last[s] = t
                hits += 1
        misses = []
        for e in U:
            if e in self.tag:
                continue
            free = [s for s in range(self.B) if self.tag[s] < 0]
            if free:
                slot = free[0]
            else:
                cand = [s for s in range(self.B) if self.last[s] < t]
                if not cand:
                    misses.append((e, -1))
                    continue
                slot = min(cand, key=lambda s: (self.last[s], self.tag[s]))
            self.tag[slot] = e
            self.last[slot] = t
            misses.append((e, slot))
        self.t += 1
        bypass = sum(1 for _, s in misses if s < 0)
        return hits, len(misses), bypass, misses


class LRUList:
    """LRU cache of B slots as a list ordered from least to most recently used.

    Within one step, the experts touched are appended in ascending id, so among experts last used
    in the same step the lower id is evicted first.
    """

    def __init__(self, E: int, B: int):
        if not (0 < B < E):
            raise ValueError("need 0 < B < E")
        self.E, self.B = E, B
        self.order = []          # experts, least recently used first
        self.slot_of = {}        # expert -> slot
        self.free = list(range(B))

    def step(self, ids):
        U = sorted(set(int(e) for e in np.asarray(ids).reshape(-1)))
        for e in U:
            if not 0 <= e < self.E:
                raise ValueError(f"expert id {e} out of range")
        touched = [e for e in U if e in self.slot_of]
        hits = len(touched)
        for e in touched:
            self.order.remove(e)
        misses = []
        for e in U:
            if e in self.slot_of:
                continue
            if self.free:
                slot = self.free.pop(0)
            elif self.order:
                victim = self.order.pop(0)
                slot = self.slot_of.pop(victim)
            else:
                misses.append((e, -1))
                continue
            self.slot_of[e] = slot
            touched.append(e)
            misses.append((e, slot))
        self.order.extend(sorted(touched))
        bypass = sum(1 for _, s in misses if s < 0)
        return hits, len(misses), bypass, misses

    def state(self):
        """(tag per slot) for comparison with LRUStamps."""
        tag = [-1] * self.B
        for e, s in self.slot_of.items():
            tag[s] = e
        return tag


def simulate(steps_ids, E: int, B: int, cls=LRUStamps):
    """Run one layer's cache over a stream of steps; steps_ids[t] holds the ids chosen at step t.

    Returns per-step arrays hits, fetches, bypass and the list of per-step miss lists.
    """
    c = cls(E, B)
    h, f, b, ml = [], [], [], []
    for ids in steps_ids:
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
