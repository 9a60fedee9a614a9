"""Pins of the oracle's batched decode step (several sequences per step; the paper describes
batch-1 decoding, the batched reading is: one lookup-table step per layer-step for the union of
the sequences' selections, each sequence's output the batch-1 MoE layer with its own routing).

Checked against: a residency-free numpy float64 evaluation per sequence, an independent
recency-list LRU fed each layer-step's union, cap invariance, a batch of identical sequences
(equal to batch 1), and sequence order (permuting the sequences permutes the outputs and leaves
the trace unchanged)."""
import numpy as np
import pytest

import oracle
import synth
from oracle.brute import RecencyListLRU

WL = synth.Workload("oracle_b4", d=128, n_experts=8, top_k=2, d_ff=128, n_layers=2, wdtype="fp32", adtype="fp32",
                    tokens=10, batch=4, rho=0.8, cap_slots=6)


@pytest.fixture(scope="module")
def setup():
    routers = [synth.router_weights(WL, l) for l in range(WL.n_layers)]
    experts = {(l, e): synth.expert_weights(WL, l, e) for l in range(WL.n_layers) for e in range(WL.n_experts)}
    hidden = synth.hidden_all(WL)  # [T x L x B x d]
    return routers, experts, hidden


def _run(setup, cap, hidden=None):
    routers, experts, hid = setup
    hid = hid if hidden is None else hidden
    orc = oracle.Oracle.for_workload(WL, cap_slots=cap, routers=routers, experts=lambda l, e: experts[(l, e)])
    res = [orc.decode_step(hid[t]) for t in range(hid.shape[0])]
    return (np.stack([r.out for r in res]), np.concatenate([r.records for r in res]), np.stack([r.idx for r in res]))


def test_each_sequence_is_the_residency_free_moe_layer(setup):
    routers, experts, hidden = setup
    out, _, idx = _run(setup, WL.cap_slots)
    for t in range(4):
        for l in range(WL.n_layers):
            Wr = np.asarray(routers[l], dtype=np.float64)
            for b in range(WL.batch):
                h = hidden[t, l, b].astype(np.float64)
                z = Wr @ h
                sel = np.lexsort((np.arange(WL.n_experts), -z))[:WL.top_k]
                assert sel.tolist() == idx[t, l, b].tolist()
                p = np.exp(z - z.max())
                g = p[sel] / p[sel].sum()
                acc = np.zeros(WL.d)
                for r, e in enumerate(sel):
                    w = experts[(l, int(e))]
                    a = w.gate.astype(np.float64) @ h
                    u = a / (1 + np.exp(-a)) * (w.up.astype(np.float64) @ h)
                    acc += g[r] * (w.down.astype(np.float64) @ u)
                np.testing.assert_allclose(out[t, l, b], acc, rtol=1e-10, atol=1e-12)


def test_trace_is_the_recency_list_over_each_layer_steps_union(setup):
    _, rec, idx = _run(setup, WL.cap_slots)
    ref = RecencyListLRU(WL.cap_slots)
    expect = []
    for t in range(idx.shape[0]):
        for l in range(WL.n_layers):
            expect += ref.step({l * WL.n_experts + int(e) for e in idx[t, l].ravel()})
    got = [(int(r["layer"]) * WL.n_experts + int(r["expert"]), int(r["kind"]), int(r["slot"]), int(r["evicted"]))
           for r in rec]
    assert got == expect
    # one record per distinct expert of the layer-step, not per sequence
    assert len(rec) == sum(len(set(idx[t, l].ravel())) for t in range(idx.shape[0]) for l in range(WL.n_layers))


def test_outputs_do_not_depend_on_the_cap(setup):
    out_a, rec_a, _ = _run(setup, WL.cap_slots)
    out_b, rec_b, _ = _run(setup, WL.n_gid)
    np.testing.assert_array_equal(out_a, out_b)
    assert (rec_a["evicted"] >= 0).sum() > 0 and (rec_b["evicted"] >= 0).sum() == 0


def test_identical_sequences_reduce_to_batch_one(setup):
    _, _, hidden = setup
    same = np.repeat(hidden[:, :, :1], WL.batch, axis=2)
    out, rec, _ = _run(setup, WL.cap_slots, hidden=same)
    for b in range(1, WL.batch):
        np.testing.assert_array_equal(out[:, :, b], out[:, :, 0])
    out1, rec1, _ = _run(setup, WL.cap_slots, hidden=np.ascontiguousarray(hidden[:, :, :1]))
    np.testing.assert_array_equal(out[:, :, 0], out1[:, :, 0])
    np.testing.assert_array_equal(rec, rec1)


def test_sequence_order_permutes_outputs_only(setup):
    _, _, hidden = setup
    perm = [2, 0, 3, 1]
    out, rec, _ = _run(setup, WL.cap_slots)
    out_p, rec_p, _ = _run(setup, WL.cap_slots, hidden=np.ascontiguousarray(hidden[:, :, perm]))
    np.testing.assert_array_equal(out_p, out[:, :, perm])
    np.testing.assert_array_equal(rec_p, rec)
