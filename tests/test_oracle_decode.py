"""Pins of the oracle's full decode step on the tiny fp32 workload (d=256, E=8, top-2,
I=128, 64 AR(1) tokens, 4 slots).

The residency cap changes only where weights are read from (paper Fig. 1: host tier vs
slot group), never the result: outputs must be bit-identical with and without the cap,
while the traces differ. Also checked: the trace equals an independent recency-list LRU
fed with the oracle's own selections, and outputs equal a residency-free numpy float64
evaluation of the MoE layer.
"""
import numpy as np
import pytest

import oracle
import synth
from oracle.brute import RecencyListLRU

WL = synth.WORKLOADS["tiny_fp32"]


@pytest.fixture(scope="module")
def tiny():
    routers = [synth.router_weights(WL, 0)]
    experts = {e: synth.expert_weights(WL, 0, e) for e in range(WL.n_experts)}
    hidden = synth.hidden_all(WL)  # [T x L x B x d]
    return routers, experts, hidden


def _run(tiny, cap, keep=True, tokens=None):
    routers, experts, hidden = tiny
    orc = oracle.Oracle.for_workload(WL, cap_slots=cap, keep_slot_copies=keep, routers=routers,
                                     experts=lambda l, e: experts[e])
    outs, recs, idxs = [], [], []
    for t in range(hidden.shape[0] if tokens is None else tokens):
        r = orc.decode_step(hidden[t])
        outs.append(r.out)
        recs.append(r.records)
        idxs.append(r.idx)
    return np.stack(outs), np.concatenate(recs), np.stack(idxs), orc


def test_outputs_identical_with_and_without_cap(tiny):
    out_cap, rec_cap, idx_cap, _ = _run(tiny, 4)
    out_all, rec_all, idx_all, _ = _run(tiny, 8)
    np.testing.assert_array_equal(out_cap, out_all)
    np.testing.assert_array_equal(idx_cap, idx_all)
    assert (rec_cap["kind"] == 1).sum() > (rec_all["kind"] == 1).sum()
    assert (rec_all["evicted"] >= 0).sum() == 0
    assert (rec_cap["evicted"] >= 0).sum() > 0


def test_slot_copies_give_the_same_bits_as_direct_reads(tiny):
    out_slots, *_ = _run(tiny, 4, keep=True, tokens=16)
    out_direct, *_ = _run(tiny, 4, keep=False, tokens=16)
    np.testing.assert_array_equal(out_slots, out_direct)


def test_trace_matches_recency_list_on_oracle_selections(tiny):
    _, rec, idx, _ = _run(tiny, 4)
    ref = RecencyListLRU(4)
    got = [(int(r["expert"]), int(r["kind"]), int(r["slot"]), int(r["evicted"])) for r in rec]
    expect = []
    for t in range(idx.shape[0]):
        expect += ref.step(idx[t, 0, 0].tolist())
    assert got == expect
    # temporal locality of the AR(1) inputs shows up as hits
    assert (rec["kind"] == 0).sum() > 0


def test_outputs_match_residency_free_numpy(tiny):
    routers, experts, hidden = tiny
    Wr = np.asarray(routers[0], dtype=np.float64)
    out, _, idx, _ = _run(tiny, 4, tokens=12)
    for t in range(12):
        h = hidden[t, 0, 0].astype(np.float64)
        z = Wr @ h
        sel = np.lexsort((np.arange(WL.n_experts), -z))[:WL.top_k]
        assert sel.tolist() == idx[t, 0, 0].tolist()
        p = np.exp(z - z.max())
        g = p[sel] / p[sel].sum()
        acc = np.zeros(WL.d)
        for r, e in enumerate(sel):
            w = experts[int(e)]
            a = w.gate.astype(np.float64) @ h
            u = a / (1 + np.exp(-a)) * (w.up.astype(np.float64) @ h)
            acc += g[r] * (w.down.astype(np.float64) @ u)
        np.testing.assert_allclose(out[t, 0, 0], acc, rtol=1e-10, atol=1e-12)


def test_a_corrupted_slot_copy_breaks_the_cap_invariant(tiny):
    """Plants a mistake in the oracle's slot storage and checks the invariant notices."""
    routers, experts, hidden = tiny
    orc = oracle.Oracle.for_workload(WL, cap_slots=4, routers=routers, experts=lambda l, e: experts[e])
    ref = oracle.Oracle.for_workload(WL, cap_slots=8, routers=routers, experts=lambda l, e: experts[e])
    orc.decode_step(hidden[0])
    ref.decode_step(hidden[0])
    gid, w = orc.slots[0]
    w.gate[0, :] *= 1.5  # a stale / wrong copy in slot 0
    diffs = 0
    for t in range(1, 8):
        a = orc.decode_step(hidden[t]).out
        b = ref.decode_step(hidden[t]).out
        diffs += int(not np.array_equal(a, b))
    assert diffs > 0


def test_step_clock_and_records_cover_every_layer_step():
    wl = WL.replace(n_layers=3, tokens=5)
    orc = oracle.Oracle.for_workload(wl, cap_slots=6)
    hidden = synth.hidden_all(wl)
    for t in range(5):
        r = orc.decode_step(hidden[t], compute_out=False)
        assert r.out is None
        assert r.records["step"].tolist() == [t] * len(r.records)
        assert sorted(set(r.records["layer"].tolist())) == [0, 1, 2]
        for l in range(3):
            got = sorted(int(e) for e in r.records[r.records["layer"] == l]["expert"])
            assert got == sorted(set(r.idx[l, 0].tolist()))
