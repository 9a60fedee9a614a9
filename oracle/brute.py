"""Pure-Python brute force for tiny inputs (test infrastructure only).

Independent restatements used to pin the C oracle, written differently on
purpose: routing sorts the full softmax explicitly; residency keeps a recency
list instead of timestamps; the expert FFN is explicit Python loops.
"""
from __future__ import annotations

import cmath
import math


def router_brute(Wr, h, k, renorm=True):
    """Full softmax over all experts, explicit sort by (-logit, id), first k, renormalise."""
    E = len(Wr)
    z = [sum(Wr[e][j] * h[j] for j in range(len(h))) for e in range(E)]
    m = max(z)
    ex = [math.exp(v - m) for v in z]
    tot = sum(ex)
    p = [v / tot for v in ex]
    order = sorted(range(E), key=lambda e: (-z[e], e))
    sel = order[:k]
    if renorm:
        s = sum(p[e] for e in sel)
        g = [p[e] / s for e in sel]
    else:
        g = [p[e] for e in sel]
    return sel, g, z, p


def expert_brute(Wg, Wu, Wd, x):
    """y = W_d (silu(W_g x) * (W_u x)) with explicit loops."""
    I, d = len(Wg), len(x)
    u = []
    for i in range(I):
        a = sum(Wg[i][j] * x[j] for j in range(d))
        b = sum(Wu[i][j] * x[j] for j in range(d))
        u.append(a / (1.0 + math.exp(-a)) * b)
    return [sum(Wd[o][i] * u[i] for i in range(I)) for o in range(len(Wd))]


class RecencyListLRU:
    """LRU over a fixed slot group kept as a recency list (oldest first).

    Residents are ordered by (time of last use, id). Each step: needed ids are
    pinned; misses (ascending id) take the lowest free slot, else the oldest
    unpinned resident's slot; then every needed id moves to the back of the
    list, in ascending id order (they share the newest use time).
    """

    def __init__(self, cap):
        self.cap = cap
        self.order = []  # resident ids, least recent first
        self.slot = {}  # id -> slot
        self.free = list(range(cap))

    def step(self, needed):
        needed = sorted(set(needed))
        pinned = set(needed)
        recs = []
        for g in needed:
            if g in self.slot:
                recs.append((g, 0, self.slot[g], -1))
                continue
            if self.free:
                s = min(self.free)
                self.free.remove(s)
                victim = -1
            else:
                victim = next((v for v in self.order if v not in pinned), None)
                if victim is None:
                    raise RuntimeError("capacity below the step's working set")
                self.order.remove(victim)
                s = self.slot.pop(victim)
            self.slot[g] = s
            recs.append((g, 1, s, victim))
        self.order = [v for v in self.order if v not in pinned] + needed
        return recs


def admit_brute(lru, needed, admit):
    """Prefetch admission on a RecencyListLRU right after its step(needed).

    Written on the recency list: ids in admit (ascending) that are absent take the lowest free
    slot, else the slot of the oldest resident outside needed and admit; when there is none the
    rest are dropped. Newly admitted ids join the needed ones at the newest use time, the group
    ordered by id. Returns records (id, 2, slot, evicted).
    """
    needed = sorted(set(needed))
    admit = sorted(set(admit))
    keep = set(needed) | set(admit)
    recs = []
    new = []
    for g in admit:
        if g in lru.slot:
            continue
        if lru.free:
            s = min(lru.free)
            lru.free.remove(s)
            victim = -1
        else:
            victim = next((v for v in lru.order if v not in keep), None)
            if victim is None:
                break
            lru.order.remove(victim)
            s = lru.slot.pop(victim)
        lru.slot[g] = s
        new.append(g)
        recs.append((g, 2, s, victim))
    newest = set(needed) | set(new)
    lru.order = [v for v in lru.order if v not in newest] + sorted(newest)
    return recs


def prefetch_candidates_brute(z, sel, m):
    """The m largest logits outside sel, by repeated arg-max with ties to the lower id."""
    left = [e for e in range(len(z)) if e not in set(sel)]
    out = []
    for _ in range(min(m, len(left))):
        best = left[0]
        for e in left[1:]:
            if z[e] > z[best]:
                best = e
        out.append(best)
        left.remove(best)
    return out


def ranks_brute(z):
    """Rank of e = how many experts beat it: a higher logit, or an equal logit and a lower id."""
    return [sum(1 for j in range(len(z)) if z[j] > z[e] or (z[j] == z[e] and j < e)) for e in range(len(z))]


class GuidedResidents:
    """Router-guided replacement kept as a dict of residents and a free list.

    The victim is chosen by comparing every evictable resident's (rank, last use, id) in one max():
    largest rank first, then the most recent use, then the lowest id. Misses in ascending id take
    the lowest free slot first; every needed id is stamped with the step counter afterwards.
    """

    def __init__(self, cap, n_experts):
        self.cap, self.E = cap, n_experts
        self.slot = {}
        self.last = {}
        self.rank = {}
        self.free = list(range(cap))
        self.t = 0

    def set_ranks(self, layer, ranks):
        for e, r in enumerate(ranks):
            self.rank[layer * self.E + e] = r

    def step(self, needed):
        needed = sorted(set(needed))
        recs = []
        for g in needed:
            if g in self.slot:
                recs.append((g, 0, self.slot[g], -1))
                continue
            if self.free:
                s = min(self.free)
                self.free.remove(s)
                victim = -1
            else:
                cands = [v for v in self.slot if v not in needed]
                if not cands:
                    raise RuntimeError("capacity below the step's working set")
                victim = max(cands, key=lambda v: (self.rank.get(v, self.E), self.last.get(v, -1), -v))
                s = self.slot.pop(victim)
            self.slot[g] = s
            recs.append((g, 1, s, victim))
        for g in needed:
            self.last[g] = self.t
        self.t += 1
        return recs


class RecencyListMRU(RecencyListLRU):
    """The recency list with the most recent evictable resident as the victim (newest first; among
    ids of the same step, the lowest id)."""

    def __init__(self, cap):
        super().__init__(cap)
        self.t = 0
        self.stamp = {}  # id -> the step it was last used in

    def step(self, needed):
        needed = sorted(set(needed))
        pinned = set(needed)
        recs = []
        for g in needed:
            if g in self.slot:
                recs.append((g, 0, self.slot[g], -1))
                continue
            if self.free:
                s = min(self.free)
                self.free.remove(s)
                victim = -1
            else:
                group = []  # the newest step's evictable ids, then older steps
                for v in reversed(self.order):
                    if v in pinned:
                        continue
                    if group and self.stamp[v] != self.stamp[group[0]]:
                        break
                    group.append(v)
                if not group:
                    raise RuntimeError("capacity below the step's working set")
                victim = min(group)
                self.order.remove(victim)
                s = self.slot.pop(victim)
            self.slot[g] = s
            recs.append((g, 1, s, victim))
        self.t += 1
        for g in needed:
            self.stamp[g] = self.t
        self.order = [v for v in self.order if v not in pinned] + needed
        return recs


class RotaryRing:
    """Independent pure-Python model of the rotary slot group (ring of slots, a hand, and each
    slot's previous occupant), for checking orc_rotary_step on random request sequences."""

    def __init__(self, cap):
        self.cap = cap
        self.ring = [None] * cap  # occupant of each slot
        self.prev = [None] * cap  # occupant evicted most recently from each slot
        self.hand = 0

    def step(self, needed):
        need = sorted(set(needed))
        pinned = set(need)
        recs = []
        for g in need:
            if g in self.ring:
                recs.append((g, 0, self.ring.index(g), -1))
                continue
            free = lambda s: self.ring[s] is None or self.ring[s] not in pinned
            back = [s for s in range(self.cap) if self.prev[s] == g and free(s)]
            if back:
                s = back[0]
            else:
                order = [(self.hand + j) % self.cap for j in range(self.cap)]
                cand = [s for s in order if free(s)]
                if not cand:
                    raise RuntimeError("no slot")
                s = cand[0]
                self.hand = (s + 1) % self.cap
            v = self.ring[s]
            self.prev = [None if p == g else p for p in self.prev]
            self.prev[s] = v
            self.ring[s] = g
            recs.append((g, 1, s, -1 if v is None else v))
        return recs


def rmsnorm_brute(x, w, eps):
    """Explicit loop: divide by the root of the mean square plus eps, then scale by w."""
    ms = sum(v * v for v in x) / len(x)
    r = math.sqrt(ms + eps)
    return [w[i] * x[i] / r for i in range(len(x))]


def rope_brute(x, pos, theta):
    """Rotary embedding as complex multiplication: the pair (x_i, x_{i+D/2}) is the complex number
    x_i + j x_{i+D/2}, multiplied by exp(j pos theta^(-2i/D))."""
    D = len(x)
    h = D // 2
    out = [0.0] * D
    for i in range(h):
        c = complex(x[i], x[i + h]) * cmath.exp(1j * pos * theta ** (-2.0 * i / D))
        out[i], out[i + h] = c.real, c.imag
    return out


def attend_brute(q, K, V, T):
    """q [Hq][D], K/V [Hkv][>=T][D]: per query head, scores over positions, a softmax written out
    with math.exp, and the weighted sum of value rows."""
    Hq, Hkv, D = len(q), len(K), len(q[0])
    out = []
    for h in range(Hq):
        g = h * Hkv // Hq
        s = [sum(q[h][i] * K[g][j][i] for i in range(D)) / math.sqrt(D) for j in range(T)]
        m = max(s)
        e = [math.exp(v - m) for v in s]
        tot = sum(e)
        out.append([sum(e[j] / tot * V[g][j][i] for j in range(T)) for i in range(D)])
    return out
