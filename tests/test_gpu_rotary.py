"""The rotary slot-group policy (MOE_POLICY_ROTARY: both batch-1 schedules, and batched steps on
both expert-FFN paths) through the C ABI against the oracle's rotary step: the residency trace
is bit-exact; outputs are within the dtype's tolerance of the fp64 oracle and bit-identical to
the LRU policy's (the policy only changes where the weights are read from)."""
import numpy as np
import pytest

import oracle
import synth
from tests.gpu_harness import TOL, check_routing, oracle_trace, rel_l2_rows, run_gpu, trace_tuples

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def P():
    import paper_2605_29135_gb300 as P

    P.build()
    return P


# "host_lookahead": the host schedule routing layer l + 1 while layer l computes. Rotary victims can
# be experts the previous layer still reads, so this also covers the copy that must wait for them.
SCHEDULES = ["device", "host_copy_engine", "host_lookahead"]


def _run(wl, cap, policy, preload=False, schedule="device", path="auto"):
    from paper_2605_29135_gb300.workload import create_for_workload

    hidden = synth.hidden_all(wl)
    look = schedule == "host_lookahead"
    m = create_for_workload(wl, cap_slots=cap, schedule="host_copy_engine" if look else schedule, policy=policy,
                            lookahead=look, batched_path=path)
    try:
        if preload:
            m.preload()
        out, idx, gate = run_gpu(m, hidden, wl.adtype)
        tr = m.get_residency_trace()
        stats = m.get_stats()
    finally:
        m.destroy()
    return hidden, out, idx, gate, tr, stats


@pytest.mark.parametrize("schedule", SCHEDULES)
@pytest.mark.parametrize("cap", [2, 3, 5])
def test_tiny_rotary_trace_and_outputs(P, cap, schedule):
    wl = synth.WORKLOADS["tiny_fp32"].replace(n_layers=2)
    hidden, out, idx, gate, tr, stats = _run(wl, cap, "rotary", schedule=schedule)
    orc = oracle.Oracle.for_workload(wl, cap_slots=cap, policy="rotary")
    res = [orc.decode_step(hidden[t], forced_idx=idx[t]) for t in range(wl.tokens)]
    np.testing.assert_array_equal(trace_tuples(tr), trace_tuples(np.concatenate([r.records for r in res])))
    assert rel_l2_rows(out, np.stack([r.out for r in res])).max() <= TOL["fp32"]
    assert stats["misses"] == int((tr["kind"] == 1).sum()) and stats["evictions"] == int((tr["evicted"] >= 0).sum())
    _, out_lru, _, _, tr_lru, _ = _run(wl, cap, "lru", schedule=schedule)
    np.testing.assert_array_equal(out, out_lru)  # same arithmetic whatever the slot contents
    if cap == 5:
        assert not np.array_equal(trace_tuples(tr), trace_tuples(tr_lru))  # the policies do differ


@pytest.mark.parametrize("schedule", SCHEDULES)
def test_rotary_preload(P, schedule):
    wl = synth.WORKLOADS["tiny_fp32"].replace(n_layers=2, tokens=32)
    hidden, out, idx, gate, tr, _ = _run(wl, 6, "rotary", preload=True, schedule=schedule)
    orc = oracle.Oracle.for_workload(wl, cap_slots=6, policy="rotary")
    orc.preload()
    recs = [orc.decode_step(hidden[t], compute_out=False, forced_idx=idx[t]).records for t in range(wl.tokens)]
    np.testing.assert_array_equal(trace_tuples(tr), trace_tuples(np.concatenate(recs)))


@pytest.mark.parametrize("schedule", SCHEDULES)
@pytest.mark.parametrize("name", ["stack48_bf16", "stack48_int4"])
def test_stack48_rotary_512_tokens(P, name, schedule):
    wl = synth.WORKLOADS[name].replace(tokens=512)
    hidden, out, idx, gate, tr, _ = _run(wl, wl.cap_slots, "rotary", schedule=schedule)
    routers = [synth.router_weights(wl, l) for l in range(wl.n_layers)]
    oidx, oz, otr = oracle_trace(wl, hidden, wl.cap_slots, routers=routers, policy="rotary")
    if check_routing(idx, oidx, oz, wl.top_k):
        _, _, otr = oracle_trace(wl, hidden, wl.cap_slots, forced_idx=idx, routers=routers, policy="rotary")
    np.testing.assert_array_equal(trace_tuples(tr), trace_tuples(otr))
    orc = oracle.Oracle.for_workload(wl, keep_slot_copies=False, routers=routers)
    for t, l in [(0, 0), (255, 20), (511, 47)]:
        ref, _, _ = orc.moe_layer(l, hidden[t, l, 0], forced_idx=idx[t, l, 0])
        assert rel_l2_rows(out[t, l, 0], ref) <= TOL[wl.wdtype]


# Batched steps: the union of the batch's experts goes through one rotary step per layer-step.
BATCHED = {
    # CUDA-core grouped GEMV: ragged fp32 shape, 4 sequences, caps that evict every step
    "fp32": synth.Workload("rb_fp32", d=256, n_experts=8, top_k=2, d_ff=128, n_layers=3, wdtype="fp32",
                           adtype="fp32", tokens=24, batch=4, rho=0.9, cap_slots=9),
    # tensor-core shape (bf16, d a multiple of 128, d_ff of 64): 66 pairs over 20 experts
    "bf16_tc": synth.Workload("rb_bf16_tc", d=384, n_experts=20, top_k=6, d_ff=192, n_layers=2, wdtype="bf16",
                              adtype="bf16", tokens=8, batch=11, rho=0.8, cap_slots=28),
    "int4": synth.Workload("rb_int4", d=384, n_experts=12, top_k=3, d_ff=256, n_layers=2, wdtype="int4",
                           adtype="bf16", tokens=10, batch=6, rho=0.8, cap_slots=14),
}


@pytest.mark.parametrize("name,path", [("fp32", "auto"), ("bf16_tc", "auto"), ("bf16_tc", "cuda_cores"),
                                       ("int4", "auto")])
def test_batched_rotary_trace_and_outputs(P, name, path):
    wl = BATCHED[name]
    hidden, out, idx, gate, tr, stats = _run(wl, wl.cap_slots, "rotary", path=path)
    routers = [synth.router_weights(wl, l) for l in range(wl.n_layers)]
    oidx, oz, otr = oracle_trace(wl, hidden, wl.cap_slots, routers=routers, policy="rotary")
    if check_routing(idx, oidx, oz, wl.top_k):
        _, _, otr = oracle_trace(wl, hidden, wl.cap_slots, forced_idx=idx, routers=routers, policy="rotary")
    np.testing.assert_array_equal(trace_tuples(tr), trace_tuples(otr))
    assert (tr["evicted"] >= 0).any()  # the cap made the ring turn
    assert stats["misses"] == int((tr["kind"] == 1).sum()) and stats["evictions"] == int((tr["evicted"] >= 0).sum())
    orc = oracle.Oracle.for_workload(wl, keep_slot_copies=False, routers=routers)
    errs = []
    for t in range(wl.tokens):
        for l in range(wl.n_layers):
            for b in range(wl.batch):
                ref, _, _ = orc.moe_layer(l, hidden[t, l, b], forced_idx=idx[t, l, b])
                errs.append(rel_l2_rows(out[t, l, b], ref))
    assert max(errs) <= TOL[wl.wdtype]
    _, out_lru, _, _, _, _ = _run(wl, wl.cap_slots, "lru", path=path)
    np.testing.assert_array_equal(out, out_lru)


def test_batched_rotary_preload(P):
    wl = BATCHED["fp32"].replace(tokens=12)
    hidden, out, idx, gate, tr, _ = _run(wl, 10, "rotary", preload=True)
    orc = oracle.Oracle.for_workload(wl, cap_slots=10, policy="rotary")
    orc.preload()
    recs = [orc.decode_step(hidden[t], compute_out=False, forced_idx=idx[t]).records for t in range(wl.tokens)]
    np.testing.assert_array_equal(trace_tuples(tr), trace_tuples(np.concatenate(recs)))


def test_stack48_batch64_rotary_capped_steps(P):
    wl = synth.WORKLOADS["stack48_batch64"].replace(tokens=3)
    hidden, out, idx, gate, tr, _ = _run(wl, wl.cap_slots, "rotary")
    routers = [synth.router_weights(wl, l) for l in range(wl.n_layers)]
    oidx, oz, otr = oracle_trace(wl, hidden, wl.cap_slots, routers=routers, policy="rotary")
    if check_routing(idx, oidx, oz, wl.top_k):
        _, _, otr = oracle_trace(wl, hidden, wl.cap_slots, forced_idx=idx, routers=routers, policy="rotary")
    np.testing.assert_array_equal(trace_tuples(tr), trace_tuples(otr))
    orc = oracle.Oracle.for_workload(wl, keep_slot_copies=False, routers=routers)
    for t, l, b in [(0, 0, 0), (1, 30, 17), (2, 47, 63)]:
        ref, _, _ = orc.moe_layer(l, hidden[t, l, b], forced_idx=idx[t, l, b])
        assert rel_l2_rows(out[t, l, b], ref) <= TOL[wl.wdtype]
