"""Pins of the oracle's prefetch admission (one reading of the paper's principle that residency
decisions may use information produced during execution, Sec. 3 and the routing result of Fig. 1):
after each layer-step's LRU step, the experts each sequence's router ranks right after its top k
are admitted into the slot group, evicting only experts the layer-step does not need.

Checked against: a hand-simulated 4-slot trace (tests/golden/lru_prefetch_hand_trace_4slot.txt),
an independent recency-list restatement on random sequences, a repeated-arg-max ranking of the
candidates, and invariants (depth 0 is plain LRU; outputs never depend on residency; admission
never evicts a needed expert; the lookup table stays a bijection).
"""
import os

import numpy as np
import pytest

import oracle
import synth
from oracle.brute import RecencyListLRU, admit_brute, prefetch_candidates_brute

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "lru_prefetch_hand_trace_4slot.txt")


def _read_golden():
    steps = {}
    for line in open(GOLDEN):
        line = line.split("#")[0].strip()
        if not line:
            continue
        lhs, rhs = line.split("|")
        s, a, b, c = (int(v) for v in lhs.split())
        e, kind, slot, ev = (int(v) for v in rhs.split())
        steps.setdefault(s, ((a, b), c, []))[2].append((e, kind, slot, ev))
    return [steps[s] for s in sorted(steps)]


def _recs(recs, E):
    return [(int(r["layer"]) * E + int(r["expert"]), int(r["kind"]), int(r["slot"]), int(r["evicted"])) for r in recs]


def test_hand_simulated_four_slot_trace():
    golden = _read_golden()
    t = oracle.LRUTable(n_gid=8, cap=4, n_experts=8)
    counts = {0: 0, 1: 0, 2: 0}
    evictions = 0
    for s, (needed, cand, expect) in enumerate(golden):
        got = _recs(t.step(clock=s, needed=needed, step=s), 8)
        got += _recs(t.admit(clock=s, pinned=needed, admit=[cand], step=s), 8)
        assert got == expect, f"step {s}"
        for g in got:
            counts[g[1]] += 1
            evictions += g[3] >= 0
    assert (counts[0], counts[1], counts[2], evictions) == (4, 8, 4, 8)
    assert t.gid_of.tolist() == [4, 2, 0, 6]


@pytest.mark.parametrize("seed", range(6))
@pytest.mark.parametrize("n_layers,E,k,m,cap", [(1, 8, 2, 1, 4), (3, 8, 2, 2, 5), (4, 16, 4, 3, 9),
                                                 (2, 32, 8, 8, 12), (2, 16, 2, 6, 7)])
def test_matches_recency_list_on_random_sequences(seed, n_layers, E, k, m, cap):
    rng = np.random.default_rng(seed)
    t = oracle.LRUTable(n_gid=n_layers * E, cap=cap, n_experts=E)
    ref = RecencyListLRU(cap)
    for tok in range(50):
        for l in range(n_layers):
            clock = tok * n_layers + l
            order = [l * E + int(e) for e in rng.permutation(E)]
            needed, cand = order[:k], order[k:k + m]
            got = _recs(t.step(clock, needed, tok), E)
            assert got == ref.step(needed), f"token {tok} layer {l}"
            got = _recs(t.admit(clock, needed, cand, tok), E)
            assert got == admit_brute(ref, needed, cand), f"token {tok} layer {l} admission"


@pytest.mark.parametrize("seed", range(4))
def test_batched_union_admission_matches_recency_list(seed):
    rng = np.random.default_rng(300 + seed)
    E, k, m, B, L, cap = 16, 3, 2, 4, 3, 15
    t = oracle.LRUTable(n_gid=L * E, cap=cap, n_experts=E)
    ref = RecencyListLRU(cap)
    for tok in range(30):
        for l in range(L):
            needed, cand = set(), set()
            for _ in range(B):
                order = [l * E + int(e) for e in rng.permutation(E)]
                needed.update(order[:k])
                cand.update(order[k:k + m])
            cand -= needed
            clock = tok * L + l
            assert _recs(t.step(clock, needed, tok), E) == ref.step(needed)
            assert _recs(t.admit(clock, needed, cand, tok), E) == admit_brute(ref, needed, cand)


def test_admission_stops_when_every_slot_is_needed():
    # cap equals the layer-step's working set: nothing may be evicted for a prefetch
    t = oracle.LRUTable(n_gid=8, cap=2, n_experts=8)
    t.step(0, [1, 5], 0)
    assert len(t.admit(0, [1, 5], [2, 3], 0)) == 0
    assert sorted(t.gid_of.tolist()) == [1, 5]
    # one free slot: the lower candidate id gets it, the other is dropped
    t = oracle.LRUTable(n_gid=8, cap=3, n_experts=8)
    t.step(0, [1, 5], 0)
    assert _recs(t.admit(0, [1, 5], [3, 2], 0), 8) == [(2, 2, 2, -1)]


def test_admitted_experts_are_protected_from_each_other():
    # two candidates, one evictable resident: the second candidate must not evict the first
    t = oracle.LRUTable(n_gid=8, cap=3, n_experts=8)
    t.step(0, [0, 1, 2], 0)
    t.step(1, [3, 4], 0)  # evicts 0 and 1; residents 2 (last use 0), 3, 4
    recs = _recs(t.admit(1, [3, 4], [6, 7], 0), 8)
    assert recs == [(6, 2, int(np.flatnonzero(t.gid_of == 6)[0]), 2)]
    assert t.slot_of[7] == -1


@pytest.mark.parametrize("seed", range(5))
def test_candidates_match_repeated_argmax_with_ties(seed):
    rng = np.random.default_rng(seed)
    E = 24
    for _ in range(40):
        z = rng.integers(-3, 4, size=E).astype(np.float64)  # many exact ties
        sel = [int(e) for e in rng.choice(E, size=4, replace=False)]
        for m in (0, 1, 3, 8, E):
            assert oracle.prefetch_candidates(z, sel, m) == prefetch_candidates_brute(list(z), sel, m)


def test_candidates_are_the_next_ranks_of_the_router():
    # with the router's own top k as the selection, the candidates are ranks k .. k + m - 1
    rng = np.random.default_rng(11)
    E, d, k, m = 16, 32, 4, 5
    Wr = rng.standard_normal((E, d))
    for _ in range(20):
        h = rng.standard_normal(d)
        idx, _, z, _ = oracle.router(Wr, h, k)
        full = np.argsort(-(Wr @ h), kind="stable")
        assert oracle.prefetch_candidates(z, idx, m) == [int(e) for e in full[k:k + m]]


WL = synth.WORKLOADS["tiny_fp32"].replace(n_layers=2, tokens=24)


@pytest.fixture(scope="module")
def hidden():
    return synth.hidden_all(WL)


def _decode(hidden, cap, prefetch, keep=True):
    kw = {} if prefetch is None else {"prefetch": prefetch}
    orc = oracle.Oracle.for_workload(WL, cap_slots=cap, keep_slot_copies=keep, **kw)
    steps = [orc.decode_step(hidden[t]) for t in range(WL.tokens)]
    return steps, orc


def test_depth_zero_is_plain_lru(hidden):
    a, _ = _decode(hidden, 5, 0)
    b, _ = _decode(hidden, 5, None)
    for x, y in zip(a, b):
        np.testing.assert_array_equal(x.records, y.records)
        np.testing.assert_array_equal(x.out, y.out)


@pytest.mark.parametrize("prefetch", [1, 2, 4])
def test_outputs_do_not_depend_on_prefetch(hidden, prefetch):
    # weights read from slots filled by admissions give the same bits as the host tier
    base, _ = _decode(hidden, 5, 0)
    got, orc = _decode(hidden, 5, prefetch)
    for x, y in zip(base, got):
        np.testing.assert_array_equal(x.out, y.out)
        np.testing.assert_array_equal(x.idx, y.idx)
    assert sum(int((s.records["kind"] == 2).sum()) for s in got) > 0
    # every resident's slot copy is the expert the lookup table names
    for s, g in enumerate(orc.table.gid_of):
        if g >= 0:
            assert orc.slots[s][0] == g


@pytest.mark.parametrize("prefetch", [1, 3])
def test_trace_matches_recency_list_on_oracle_routing(hidden, prefetch):
    steps, _ = _decode(hidden, 5, prefetch, keep=False)
    E, L = WL.n_experts, WL.n_layers
    ref = RecencyListLRU(5)
    for t, st in enumerate(steps):
        expect = []
        for l in range(L):
            needed = sorted({l * E + int(e) for e in st.idx[l].ravel()})
            expect += ref.step(needed)
            cand = set()
            for b in range(st.idx.shape[1]):
                cand.update(l * E + e for e in prefetch_candidates_brute(list(st.z[l, b]), list(st.idx[l, b]), prefetch))
            expect += admit_brute(ref, needed, sorted(cand - set(needed)))
        assert _recs(st.records, E) == expect, f"token {t}"


def test_admission_never_evicts_a_needed_expert(hidden):
    steps, _ = _decode(hidden, 4, 2, keep=False)
    E = WL.n_experts
    for st in steps:
        for l in range(WL.n_layers):
            needed = {l * E + int(e) for e in st.idx[l].ravel()}
            for r in st.records[st.records["layer"] == l]:
                if r["kind"] == 2:
                    assert int(r["evicted"]) not in needed
                    assert l * E + int(r["expert"]) not in needed
