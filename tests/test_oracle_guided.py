"""Pins of the oracle's router-guided replacement (one reading of the paper's residency decisions
that use information produced during execution, Sec. 3, with the routing result of Fig. 1 as
that information): a miss evicts the resident with the largest rank in its layer's most recent
routing, ties to the more recent use, then to the lower global id.

Checked against: hand-simulated traces (tests/golden/guided_hand_trace.txt: a single layer where
the rule departs from LRU, equal ranks across layers, preloaded ties), an independent
dict-of-residents restatement on random, multi-layer, batched and preloaded sequences, the ranking
against a count-the-winners definition, and invariants (with every rank equal the rule is
most-recently-used replacement, checked against a recency list; outputs do not depend on the
policy).
"""
import os

import numpy as np
import pytest

import oracle
import synth
from oracle.brute import GuidedResidents, RecencyListMRU, ranks_brute

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "guided_hand_trace.txt")


def read_guided_golden(path=GOLDEN):
    """-> {case: (E, L, k, cap, preload, [((t, l, order), [(expert, kind, slot, evicted)])])}"""
    cases = {}
    cur = None
    for line in open(path):
        line = line.split("#")[0].strip()
        if not line:
            continue
        if line.startswith("@case"):
            _, name, E, L, k, cap, start = line.split()
            cur = cases[name] = (int(E), int(L), int(k), int(cap), start == "preload", [])
            continue
        lhs, rhs = line.split("|")
        v = [int(x) for x in lhs.split()]
        key = (v[0], v[1], tuple(v[2:]))
        steps = cur[5]
        if not steps or steps[-1][0] != key:
            steps.append((key, []))
        steps[-1][1].append(tuple(int(x) for x in rhs.split()))
    return cases


def _ranks_of(order):
    r = np.empty(len(order), dtype=np.int32)
    r[list(order)] = np.arange(len(order))
    return r


def _tuples(recs, E):
    return [(int(r["layer"]) * E + int(r["expert"]), int(r["kind"]), int(r["slot"]), int(r["evicted"])) for r in recs]


@pytest.mark.parametrize("case", ["A", "B", "C"])
def test_hand_simulated_traces(case):
    E, L, k, cap, preload, steps = read_guided_golden()[case]
    t = oracle.GuidedTable(n_gid=L * E, cap=cap, n_experts=E)
    if preload:
        t.preload()
    for (tok, l, order), expect in steps:
        t.set_layer_ranks(l, _ranks_of(order))
        needed = [l * E + e for e in order[:k]]
        recs = t.step(tok * L + l, needed, tok)
        got = [(int(r["expert"]), int(r["kind"]), int(r["slot"]), int(r["evicted"])) for r in recs]
        assert got == expect, f"case {case} token {tok} layer {l}"
        assert all(int(r["layer"]) == l for r in recs)
    final = {"A": [6, 3, 4, 2], "B": [1, 6, 0]}
    if case in final:
        assert t.gid_of.tolist() == final[case]


def _random_run(seed, n_layers, E, k, cap, B, tokens, preload=False):
    rng = np.random.default_rng(seed)
    t = oracle.GuidedTable(n_gid=n_layers * E, cap=cap, n_experts=E)
    ref = GuidedResidents(cap, E)
    if preload:
        t.preload()
        for s in range(min(cap, n_layers * E)):
            ref.slot[s] = s
            ref.last[s] = -1
            ref.free.remove(s)
    for tok in range(tokens):
        for l in range(n_layers):
            needed, best = set(), np.full(E, E, dtype=np.int32)
            for _ in range(B):
                order = [int(e) for e in rng.permutation(E)]
                needed.update(l * E + e for e in order[:k])
                best = np.minimum(best, _ranks_of(order))
            t.set_layer_ranks(l, best)
            ref.set_ranks(l, best.tolist())
            got = _tuples(t.step(tok * n_layers + l, needed, tok), E)
            assert got == ref.step(needed), f"token {tok} layer {l}"
    return t


@pytest.mark.parametrize("seed", range(5))
@pytest.mark.parametrize("n_layers,E,k,cap,B", [(1, 8, 2, 4, 1), (3, 8, 2, 5, 1), (4, 16, 4, 9, 1),
                                                (2, 32, 8, 12, 1), (3, 4, 1, 5, 1), (3, 16, 3, 14, 4)])
def test_matches_independent_residents_on_random_sequences(seed, n_layers, E, k, cap, B):
    _random_run(seed, n_layers, E, k, cap, B, 40)


@pytest.mark.parametrize("seed", range(3))
def test_matches_independent_residents_after_preload(seed):
    _random_run(70 + seed, 3, 4, 1, 7, 1, 30, preload=True)


@pytest.mark.parametrize("seed", range(4))
def test_equal_ranks_reduce_to_mru(seed):
    # every rank equal: the victim is the most recent evictable resident, then the lower id
    rng = np.random.default_rng(seed)
    E, L, k, cap = 8, 3, 2, 5
    t = oracle.GuidedTable(n_gid=L * E, cap=cap, n_experts=E)
    ref = RecencyListMRU(cap)
    for tok in range(40):
        for l in range(L):
            needed = [l * E + int(e) for e in rng.choice(E, size=k, replace=False)]
            t.set_layer_ranks(l, np.zeros(E, dtype=np.int32))
            assert _tuples(t.step(tok * L + l, needed, tok), E) == ref.step(needed)


@pytest.mark.parametrize("seed", range(5))
def test_ranks_match_count_of_winners_with_ties(seed):
    rng = np.random.default_rng(seed)
    for _ in range(30):
        z = rng.integers(-3, 4, size=16).astype(np.float64)
        assert oracle.route_ranks(z).tolist() == ranks_brute(list(z))


def test_capacity_below_working_set_is_an_error():
    t = oracle.GuidedTable(n_gid=8, cap=2, n_experts=8)
    t.set_layer_ranks(0, np.arange(8))
    with pytest.raises(RuntimeError):
        t.step(0, [1, 2, 3], 0)


WL = synth.WORKLOADS["tiny_fp32"].replace(n_layers=3, tokens=20)


def test_outputs_do_not_depend_on_the_policy():
    hidden = synth.hidden_all(WL)
    outs = []
    for policy in ("lru", "guided"):
        orc = oracle.Oracle.for_workload(WL, cap_slots=8, policy=policy)
        outs.append(np.stack([orc.decode_step(hidden[t]).out for t in range(WL.tokens)]))
    np.testing.assert_array_equal(outs[0], outs[1])


def test_decode_trace_matches_independent_residents_on_oracle_routing():
    hidden = synth.hidden_all(WL)
    E, L, cap = WL.n_experts, WL.n_layers, 8
    orc = oracle.Oracle.for_workload(WL, cap_slots=cap, policy="guided", keep_slot_copies=False)
    ref = GuidedResidents(cap, E)
    differs_from_lru = False
    lru = oracle.Oracle.for_workload(WL, cap_slots=cap, keep_slot_copies=False)
    for t in range(WL.tokens):
        st = orc.decode_step(hidden[t], compute_out=False)
        expect = []
        for l in range(L):
            ref.set_ranks(l, ranks_brute(list(st.z[l, 0])))
            expect += ref.step({l * E + int(e) for e in st.idx[l, 0]})
        assert _tuples(st.records, E) == expect, f"token {t}"
        differs_from_lru |= _tuples(lru.decode_step(hidden[t], compute_out=False).records, E) != expect
    assert differs_from_lru
