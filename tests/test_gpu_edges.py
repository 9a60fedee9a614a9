"""Edge cases of the decode step through the C ABI, against the fp64 oracle on the same inputs:
top-k equal to the expert count, router logits that tie exactly (duplicated router rows: the
lower expert id must win on the device as in the oracle), gates without renormalisation, a pool
exactly as large as one step's working set, the largest batched step (64 sequences x top-16 =
1024 routed pairs), and requests the boundary rejects. Every case runs both batch-1 schedules or
both batched expert-FFN paths."""
import numpy as np
import pytest

import oracle
import synth
from tests.gpu_harness import TOL, check_routing, rel_l2_rows, run_gpu, trace_tuples

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def P():
    import paper_2605_29135_gb300 as P

    P.build()
    return P


def _run(wl, cap, routers=None, renorm=True, schedule="device", path="auto"):
    from paper_2605_29135_gb300.workload import create_for_workload

    hidden = synth.hidden_all(wl)
    m = create_for_workload(wl, cap_slots=cap, schedule=schedule, batched_path=path, renorm=renorm)
    try:
        if routers is not None:
            for l, w in enumerate(routers):
                m.set_router(l, w)
        out, idx, gate = run_gpu(m, hidden, wl.adtype)
        tr = m.get_residency_trace()
    finally:
        m.destroy()
    return hidden, out, idx, gate, tr


def _oracle(wl, cap, hidden, routers=None, renorm=True, forced=None):
    orc = oracle.Oracle.for_workload(wl, cap_slots=cap, routers=routers, renorm=renorm)
    res = [orc.decode_step(hidden[t], forced_idx=None if forced is None else forced[t]) for t in range(wl.tokens)]
    return (np.stack([r.out for r in res]), np.stack([r.idx for r in res]), np.stack([r.gate for r in res]),
            np.stack([r.z for r in res]), np.concatenate([r.records for r in res]))


def _check(wl, cap, hidden, out, idx, gate, tr, routers=None, renorm=True, exact_ids=False):
    ref, oidx, ogate, oz, otr = _oracle(wl, cap, hidden, routers, renorm)
    if exact_ids:
        np.testing.assert_array_equal(idx, oidx)
    elif check_routing(idx, oidx, oz, wl.top_k):
        ref, oidx, ogate, oz, otr = _oracle(wl, cap, hidden, routers, renorm, forced=idx)
    np.testing.assert_array_equal(trace_tuples(tr), trace_tuples(otr))
    np.testing.assert_allclose(gate, ogate, rtol=2e-5, atol=1e-6)
    assert rel_l2_rows(out, ref).max() <= TOL[wl.wdtype]


# (schedule, batched expert-FFN path, batched?): both batch-1 schedules, both batched paths
CASES = [("device", "auto", False), ("host_copy_engine", "auto", False), ("device", "auto", True),
         ("device", "cuda_cores", True)]
IDS = ["b1-device", "b1-host_copy_engine", "batched-tensor_cores", "batched-cuda_cores"]


@pytest.mark.parametrize("schedule,path,batched", CASES, ids=IDS)
def test_top_k_equals_expert_count(P, schedule, path, batched):
    batch = 5 if batched else 1
    wl = synth.Workload("edge_k_eq_e", d=256, n_experts=4, top_k=4, d_ff=128, n_layers=2, wdtype="bf16",
                        adtype="bf16", tokens=8, batch=batch, rho=0.8, cap_slots=6)
    hidden, out, idx, gate, tr = _run(wl, wl.cap_slots, schedule=schedule, path=path)
    assert (np.sort(idx, axis=-1) == np.arange(4)).all()
    _check(wl, wl.cap_slots, hidden, out, idx, gate, tr)


def _tied_routers(wl):
    # rows 2, 9 and 13 identical and dominant (the top three ranks tie: ids must come out as 2, 9, 13);
    # rows 5 and 6 identical and moderate (they tie at the k-th rank from time to time)
    rng = np.random.default_rng(3)
    routers = []
    for _ in range(wl.n_layers):
        w = (rng.standard_normal((wl.n_experts, wl.d)) / np.sqrt(wl.d)).astype(np.float32)
        w[[2, 9, 13]] = 4.0 * w[2]
        w[6] = w[5]
        routers.append(np.ascontiguousarray(w if wl.router_dtype == "fp32" else synth.f32_to_bf16_bits(w)))
    return routers


@pytest.mark.parametrize("schedule,path,batched", CASES, ids=IDS)
def test_exactly_tied_logits_break_to_the_lower_id(P, schedule, path, batched):
    batch = 3 if batched else 1
    dt = "bf16" if batched else "fp32"  # bf16 so that the batched tensor-core path takes it
    wl = synth.Workload("edge_ties", d=256, n_experts=16, top_k=4, d_ff=128, n_layers=2, wdtype=dt,
                        adtype=dt, tokens=12, batch=batch, rho=0.8, cap_slots=12)
    routers = _tied_routers(wl)
    hidden, out, idx, gate, tr = _run(wl, wl.cap_slots, routers=routers, schedule=schedule, path=path)
    # whenever the dominant group is selected it appears in id order, with equal gates
    for pos in np.ndindex(*idx.shape[:-1]):
        sel = idx[pos].tolist()
        grp = [e for e in sel if e in (2, 9, 13)]
        assert grp == sorted(grp)
        if 5 in sel and 6 in sel:
            assert sel.index(5) < sel.index(6)
    _check(wl, wl.cap_slots, hidden, out, idx, gate, tr, routers=routers, exact_ids=True)


@pytest.mark.parametrize("schedule,path,batched", CASES, ids=IDS)
def test_gates_without_renormalisation(P, schedule, path, batched):
    batch = 4 if batched else 1
    wl = synth.Workload("edge_norenorm", d=256, n_experts=12, top_k=3, d_ff=128, n_layers=2, wdtype="bf16",
                        adtype="bf16", tokens=8, batch=batch, rho=0.8, cap_slots=14)
    hidden, out, idx, gate, tr = _run(wl, wl.cap_slots, renorm=False, schedule=schedule, path=path)
    assert (gate.sum(-1) < 1.0).all()
    _check(wl, wl.cap_slots, hidden, out, idx, gate, tr, renorm=False)


@pytest.mark.parametrize("schedule", ["device", "host_copy_engine"])
def test_pool_exactly_one_working_set(P, schedule):
    # cap = k at batch 1: every miss must evict, and only the previous layer-step's experts are resident
    wl = synth.WORKLOADS["tiny_fp32"].replace(n_layers=2, tokens=24)
    hidden, out, idx, gate, tr = _run(wl, wl.top_k, schedule=schedule)
    assert (tr["evicted"] >= 0).sum() > 0
    _check(wl, wl.top_k, hidden, out, idx, gate, tr)


@pytest.mark.parametrize("path", ["auto", "cuda_cores"])
def test_largest_batched_step(P, path):
    # 64 sequences x top-16 = 1024 routed pairs per layer-step, ~32 per expert
    wl = synth.Workload("edge_max_pairs", d=256, n_experts=32, top_k=16, d_ff=128, n_layers=2, wdtype="bf16",
                        adtype="bf16", tokens=3, batch=64, rho=0.8, cap_slots=40)
    hidden, out, idx, gate, tr = _run(wl, wl.cap_slots, path=path)
    _check(wl, wl.cap_slots, hidden, out, idx, gate, tr)


def test_boundary_rejects_bad_requests(P):
    import ctypes

    import torch

    from paper_2605_29135_gb300.workload import create_for_workload

    wl = synth.WORKLOADS["tiny_fp32"].replace(batch=4)
    m = create_for_workload(wl, cap_slots=8)
    try:
        h = torch.zeros((wl.n_layers, 4, wl.d), dtype=torch.float32, device="cuda")
        o = torch.empty_like(h)
        ptr = ctypes.c_void_p
        assert m.lib.moe_decode_step(m.h, ptr(h.data_ptr()), ptr(o.data_ptr()), 0, None) == -1  # batch 0
        assert m.lib.moe_decode_step(m.h, None, ptr(o.data_ptr()), 1, None) == -1  # NULL hidden
        assert m.lib.moe_decode_step(m.h, ptr(h.data_ptr()), None, 1, None) == -1  # NULL out
        # misaligned activation buffers are refused before any launch (one fp32 element off)
        assert m.lib.moe_decode_step(m.h, ptr(h.data_ptr() + 4), ptr(o.data_ptr()), 1, None) == -1
        assert m.lib.moe_decode_step(m.h, ptr(h.data_ptr()), ptr(o.data_ptr() + 4), 1, None) == -1
        assert m.get_stats()["layer_steps"] == 0  # nothing ran
        m.decode_step(h, o, batch=4)  # the handle still works
        torch.cuda.synchronize()
        assert m.get_stats()["layer_steps"] == wl.n_layers
    finally:
        m.destroy()
