"""The rotary slot-group policy (MOE_POLICY_ROTARY, both batch-1 schedules) through the C ABI
against the oracle's rotary step: the residency trace is bit-exact; outputs are within the
dtype's tolerance of the fp64 oracle and bit-identical to the LRU policy's (the policy only
changes where the weights are read from)."""
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


def _run(wl, cap, policy, preload=False, schedule="device"):
    from paper_2605_29135_gb300.workload import create_for_workload

    hidden = synth.hidden_all(wl)
    look = schedule == "host_lookahead"
    m = create_for_workload(wl, cap_slots=cap, schedule="host_copy_engine" if look else schedule, policy=policy,
                            lookahead=look)
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
