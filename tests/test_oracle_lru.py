"""Pins of the oracle's residency step (paper Fig. 1: slot group, lookup table, evict;
the undisclosed rotary policy replaced by deterministic LRU with lower-id ties).

Checked against: a hand-simulated 4-slot trace (tests/golden/lru_hand_trace_4slot.txt)
and an independent recency-list implementation on random request sequences.
"""
import os

import numpy as np
import pytest

import oracle
from oracle.brute import RecencyListLRU

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "lru_hand_trace_4slot.txt")


def _read_golden():
    steps = {}
    for line in open(GOLDEN):
        line = line.split("#")[0].strip()
        if not line:
            continue
        lhs, rhs = line.split("|")
        s, a, b = (int(v) for v in lhs.split())
        e, kind, slot, ev = (int(v) for v in rhs.split())
        steps.setdefault(s, ((a, b), []))[1].append((e, kind, slot, ev))
    return [steps[s] for s in sorted(steps)]


def test_hand_simulated_four_slot_trace():
    golden = _read_golden()
    t = oracle.LRUTable(n_gid=8, cap=4, n_experts=8)
    hits = misses = evictions = 0
    for s, (needed, expect) in enumerate(golden):
        recs = t.step(clock=s, needed=needed, step=s)
        got = [(int(r["expert"]), int(r["kind"]), int(r["slot"]), int(r["evicted"])) for r in recs]
        assert got == expect, f"step {s}"
        assert all(int(r["step"]) == s and int(r["layer"]) == 0 for r in recs)
        hits += sum(1 for g in got if g[1] == 0)
        misses += sum(1 for g in got if g[1] == 1)
        evictions += sum(1 for g in got if g[3] >= 0)
    assert (hits, misses, evictions) == (3, 9, 5)
    assert t.gid_of.tolist() == [2, 7, 3, 0]


@pytest.mark.parametrize("seed", range(8))
@pytest.mark.parametrize("n_layers,E,k,cap", [(1, 8, 2, 4), (3, 8, 2, 5), (4, 16, 4, 9), (2, 32, 8, 8)])
def test_matches_recency_list_on_random_sequences(seed, n_layers, E, k, cap):
    rng = np.random.default_rng(seed)
    t = oracle.LRUTable(n_gid=n_layers * E, cap=cap, n_experts=E)
    ref = RecencyListLRU(cap)
    for tok in range(60):
        for l in range(n_layers):
            clock = tok * n_layers + l
            needed = [l * E + int(e) for e in rng.choice(E, size=k, replace=False)]
            got = [(int(r["layer"]) * E + int(r["expert"]), int(r["kind"]), int(r["slot"]), int(r["evicted"]))
                   for r in t.step(clock, needed, tok)]
            assert got == ref.step(needed), f"token {tok} layer {l}"


@pytest.mark.parametrize("seed", range(4))
def test_batched_union_steps_match_recency_list(seed):
    # several sequences per layer-step: the needed set is the union of their selections
    rng = np.random.default_rng(100 + seed)
    E, k, B, L, cap = 16, 3, 4, 3, 14
    t = oracle.LRUTable(n_gid=L * E, cap=cap, n_experts=E)
    ref = RecencyListLRU(cap)
    for tok in range(30):
        for l in range(L):
            needed = {l * E + int(e) for _ in range(B) for e in rng.choice(E, size=k, replace=False)}
            got = [(int(r["layer"]) * E + int(r["expert"]), int(r["kind"]), int(r["slot"]), int(r["evicted"]))
                   for r in t.step(tok * L + l, needed, tok)]
            assert got == ref.step(needed)


def test_state_is_a_consistent_bijection():
    rng = np.random.default_rng(7)
    E, L, cap = 8, 3, 6
    t = oracle.LRUTable(n_gid=L * E, cap=cap, n_experts=E)
    for tok in range(40):
        for l in range(L):
            t.step(tok * L + l, [l * E + int(e) for e in rng.choice(E, 2, replace=False)], tok)
            for s, g in enumerate(t.gid_of):
                if g >= 0:
                    assert t.slot_of[g] == s
            assert (t.slot_of >= 0).sum() == (t.gid_of >= 0).sum()


def test_capacity_below_working_set_is_an_error():
    t = oracle.LRUTable(n_gid=8, cap=2, n_experts=8)
    t.step(0, [0, 1], 0)
    with pytest.raises(RuntimeError):
        t.step(1, [2, 3, 4], 1)


def test_cap_at_least_all_experts_never_evicts():
    t = oracle.LRUTable(n_gid=8, cap=8, n_experts=8)
    rng = np.random.default_rng(1)
    seen = set()
    for s in range(50):
        needed = [int(e) for e in rng.choice(8, 2, replace=False)]
        for r in t.step(s, needed, s):
            assert r["evicted"] == -1
            assert r["kind"] == (0 if int(r["expert"]) in seen else 1)
        seen.update(needed)


def test_preload_fills_free_slots_in_id_order_and_ages_them_first():
    # 4 slots, 8 experts: preload puts experts 0..3 in slots 0..3 with last use -1; a step needing
    # {5, 6} then misses twice and evicts 0 and 1 (oldest, lower id first); a step needing {2, 7}
    # hits 2 and evicts 3 (still last use -1) for 7.
    t = oracle.LRUTable(n_gid=8, cap=4, n_experts=8)
    t.preload()
    assert t.gid_of.tolist() == [0, 1, 2, 3]
    got = [(int(r["expert"]), int(r["kind"]), int(r["slot"]), int(r["evicted"])) for r in t.step(0, [5, 6], 0)]
    assert got == [(5, 1, 0, 0), (6, 1, 1, 1)]
    got = [(int(r["expert"]), int(r["kind"]), int(r["slot"]), int(r["evicted"])) for r in t.step(1, [2, 7], 1)]
    assert got == [(2, 0, 2, -1), (7, 1, 3, 3)]


def test_preload_with_cap_at_least_all_experts_makes_every_request_a_hit():
    t = oracle.LRUTable(n_gid=6, cap=8, n_experts=6)
    t.preload()
    assert sorted(int(g) for g in t.gid_of if g >= 0) == list(range(6))
    for s in range(5):
        assert all(int(r["kind"]) == 0 for r in t.step(s, [s % 6, (s + 3) % 6], s))
