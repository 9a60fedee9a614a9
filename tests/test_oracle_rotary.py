"""Pins of the oracle's rotary slot-group step (one reading of the paper's rotary
residency, Fig. 1 "Rotary Slot Group" and Fig. 2 "cyclical forward and reverse rotation").

Checked against: a hand-simulated 4-slot trace (tests/golden/rotary_hand_trace_4slot.txt), an
independent pure-Python ring on random request sequences, and invariants (the lookup table stays a
bijection; with the cap at least the number of experts nothing is ever evicted)."""
import os

import numpy as np
import pytest

import oracle
from oracle.brute import RotaryRing

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "rotary_hand_trace_4slot.txt")


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


def _recs(recs, E):
    return [(int(r["layer"]) * E + int(r["expert"]), int(r["kind"]), int(r["slot"]), int(r["evicted"])) for r in recs]


def test_hand_simulated_four_slot_trace():
    golden = _read_golden()
    t = oracle.RotaryTable(n_gid=8, cap=4, n_experts=8)
    counts = [0, 0, 0]
    for s, (needed, expect) in enumerate(golden):
        got = _recs(t.step(clock=s, needed=needed, step=s), 8)
        assert got == expect, f"step {s}"
        counts[0] += sum(1 for g in got if g[1] == 0)
        counts[1] += sum(1 for g in got if g[1] == 1)
        counts[2] += sum(1 for g in got if g[3] >= 0)
    assert counts == [6, 14, 10]
    assert t.gid_of.tolist() == [1, 7, 4, 0]
    assert t.prior.tolist() == [-1, 5, 2, 6]


@pytest.mark.parametrize("seed", range(6))
@pytest.mark.parametrize("n_layers,E,k,cap", [(1, 8, 2, 4), (3, 8, 2, 5), (4, 16, 4, 9), (2, 32, 8, 8)])
def test_matches_independent_ring_on_random_sequences(seed, n_layers, E, k, cap):
    rng = np.random.default_rng(seed)
    t = oracle.RotaryTable(n_gid=n_layers * E, cap=cap, n_experts=E)
    ref = RotaryRing(cap)
    for tok in range(60):
        for l in range(n_layers):
            needed = [l * E + int(e) for e in rng.choice(E, size=k, replace=False)]
            assert _recs(t.step(tok * n_layers + l, needed, tok), E) == ref.step(needed), f"token {tok} layer {l}"


@pytest.mark.parametrize("seed", range(3))
def test_batched_union_steps_match_independent_ring(seed):
    rng = np.random.default_rng(50 + seed)
    E, k, B, L, cap = 16, 3, 4, 3, 14
    t = oracle.RotaryTable(n_gid=L * E, cap=cap, n_experts=E)
    ref = RotaryRing(cap)
    for tok in range(30):
        for l in range(L):
            needed = {l * E + int(e) for _ in range(B) for e in rng.choice(E, size=k, replace=False)}
            assert _recs(t.step(tok * L + l, needed, tok), E) == ref.step(needed)


def test_state_stays_a_bijection_and_priors_are_not_resident():
    rng = np.random.default_rng(7)
    E, L, cap = 8, 3, 6
    t = oracle.RotaryTable(n_gid=L * E, cap=cap, n_experts=E)
    for tok in range(40):
        for l in range(L):
            t.step(tok * L + l, [l * E + int(e) for e in rng.choice(E, 2, replace=False)], tok)
            for s, g in enumerate(t.gid_of):
                if g >= 0:
                    assert t.slot_of[g] == s
            assert (t.slot_of >= 0).sum() == (t.gid_of >= 0).sum()
            for p in t.prior:
                assert p < 0 or t.slot_of[p] < 0  # a previous occupant is never resident
            assert len([p for p in t.prior if p >= 0]) == len({p for p in t.prior if p >= 0})


def test_cap_at_least_all_experts_never_evicts():
    t = oracle.RotaryTable(n_gid=8, cap=8, n_experts=8)
    rng = np.random.default_rng(1)
    for s in range(50):
        for r in t.step(s, [int(e) for e in rng.choice(8, 2, replace=False)], s):
            assert r["evicted"] == -1


def test_capacity_below_working_set_is_an_error():
    t = oracle.RotaryTable(n_gid=8, cap=2, n_experts=8)
    with pytest.raises(RuntimeError):
        t.step(0, [1, 2, 3], 0)


def test_outputs_do_not_depend_on_the_policy():
    # residency only changes where weights are read from: the rotary and LRU oracles give
    # bit-identical outputs on the same inputs
    import synth

    wl = synth.WORKLOADS["tiny_fp32"].replace(n_layers=2, tokens=12)
    hidden = synth.hidden_all(wl)
    outs = []
    for policy in ("lru", "rotary"):
        orc = oracle.Oracle.for_workload(wl, cap_slots=5, policy=policy)
        outs.append(np.stack([orc.decode_step(hidden[t]).out for t in range(wl.tokens)]))
    np.testing.assert_array_equal(outs[0], outs[1])
