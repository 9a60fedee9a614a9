"""Failure paths through the C ABI, exercised without faulting a GPU:

- a device-side wait that runs out: an injected fault makes a step's grid barriers wait for an
  arrival count nothing reaches; the bounded waits expire (0.2 s), the kernel exits, the host
  reports MOE_ERR_TIMEOUT and empties the pool, and the handle keeps working (the next steps
  match the oracle from a cold pool);
- a miss copy that fails (host-side shim in the copy-engine schedule): MOE_ERR_CUDA, pool
  emptied, handle keeps working;
- experts not registered: MOE_ERR_NOT_REGISTERED before any work;
- a cap below one layer-step's working set: MOE_ERR_CAPACITY at create;
- a pool larger than the device: MOE_ERR_OOM at create, nothing left allocated.
"""
import numpy as np
import pytest

import oracle
import synth
from tests.gpu_harness import TOL, rel_l2_rows, run_gpu, trace_tuples

pytestmark = pytest.mark.gpu

ERR = {"invalid": -1, "oom": -2, "cuda": -3, "capacity": -4, "not_registered": -5, "timeout": -6}


@pytest.fixture(scope="module")
def P():
    import paper_2605_29135_gb300 as P

    P.build()
    return P


def _expect_recovery(m, wl, hidden, cap):
    """After a failed step the pool is empty: the following steps reproduce the oracle's trace
    from a cold pool (step indices restart at 0)."""
    out, idx, _ = run_gpu(m, hidden, wl.adtype)
    tr = m.get_residency_trace()
    orc = oracle.Oracle.for_workload(wl, cap_slots=cap)
    res = [orc.decode_step(hidden[t], forced_idx=idx[t]) for t in range(hidden.shape[0])]
    np.testing.assert_array_equal(trace_tuples(tr), trace_tuples(np.concatenate([r.records for r in res])))
    assert rel_l2_rows(out, np.stack([r.out for r in res])).max() <= TOL[wl.wdtype]


@pytest.mark.parametrize("batch,lookahead,dtype", [(1, False, "fp32"), (4, False, "fp32"), (1, True, "fp32"),
                                                   (1, True, "bf16")])
def test_device_wait_that_runs_out_reports_timeout_and_recovers(P, batch, lookahead, dtype):
    # lookahead: the device schedule's lookahead kernel, whose router-phase barrier is the one
    # that runs out; every CTA leaves it, so no worker waits for a plan that never comes (bf16:
    # its bulk-copy variant, whose warps have issued no copies yet when they leave)
    import torch

    from paper_2605_29135_gb300.workload import create_for_workload

    wl = synth.WORKLOADS["tiny_fp32"].replace(n_layers=2, tokens=8, batch=batch)
    if dtype == "bf16":
        wl = wl.replace(wdtype="bf16", adtype="bf16")
    hidden = synth.hidden_all(wl)
    m = create_for_workload(wl, cap_slots=8, lookahead=lookahead)
    try:
        if dtype == "bf16":
            h = torch.from_numpy(hidden[0].view(np.int16)).cuda().view(torch.bfloat16)
        else:
            h = torch.from_numpy(hidden[0].view(np.float32)).cuda()
        o = torch.empty_like(h)
        m.decode_step(h, o, batch=batch)  # a normal step first
        m.inject_fault("barrier_timeout")
        m.decode_step(h, o, batch=batch)  # enqueued; the failure surfaces at the next synchronising call
        with pytest.raises(P.MoEError) as ei:
            m.get_stats()
        assert ei.value.status == ERR["timeout"]
        assert "barrier" in str(ei.value)
        st = m.get_stats()  # the flag was consumed and the state reset
        assert st["layer_steps"] == 0 and st["misses"] == 0
        _expect_recovery(m, wl, hidden, 8)
    finally:
        m.destroy()


def test_failed_miss_copy_reports_cuda_error_and_recovers(P):
    import torch

    from paper_2605_29135_gb300.workload import create_for_workload

    wl = synth.WORKLOADS["tiny_fp32"].replace(n_layers=2, tokens=8)
    hidden = synth.hidden_all(wl)
    m = create_for_workload(wl, schedule="host_copy_engine")
    try:
        h = torch.from_numpy(hidden[0].view(np.float32)).cuda()
        o = torch.empty_like(h)
        m.inject_fault("copy_error")
        with pytest.raises(P.MoEError) as ei:
            m.decode_step(h, o)
        assert ei.value.status == ERR["cuda"] and "injected" in str(ei.value)
        assert m.get_stats()["layer_steps"] == 0
        _expect_recovery(m, wl, hidden, wl.cap_slots)
    finally:
        m.destroy()


def test_fault_kinds_are_checked_against_the_schedule(P):
    from paper_2605_29135_gb300.workload import create_for_workload

    wl = synth.WORKLOADS["tiny_fp32"].replace(tokens=2)
    for schedule, bad in (("device", "copy_error"), ("host_copy_engine", "barrier_timeout")):
        m = create_for_workload(wl, schedule=schedule)
        try:
            with pytest.raises(P.MoEError) as ei:
                m.inject_fault(bad)
            assert ei.value.status == ERR["invalid"]
        finally:
            m.destroy()


@pytest.mark.parametrize("schedule", ["device", "host_copy_engine"])
def test_unregistered_expert_is_reported_before_any_work(P, schedule):
    import torch

    wl = synth.WORKLOADS["tiny_fp32"]
    cfg = P.make_config(wl.d, wl.n_experts, wl.top_k, wl.d_ff, wl.n_layers, wl.wdtype, wl.adtype, cap_slots=4,
                        schedule=schedule)
    m = P.MoE(cfg)
    try:
        m.set_router(0, synth.router_weights(wl, 0))
        for e in range(wl.n_experts):
            if e == 5:
                continue  # expert 5 of layer 0 never registered
            w = synth.expert_weights(wl, 0, e)
            m.register_host_experts(0, e, w.gate, w.up, w.down, w.scales_flat())
        h = torch.zeros((1, 1, wl.d), dtype=torch.float32, device="cuda")
        with pytest.raises(P.MoEError) as ei:
            m.decode_step(h, torch.empty_like(h))
        assert ei.value.status == ERR["not_registered"] and "expert 5 of layer 0" in str(ei.value)
        assert m.get_stats()["layer_steps"] == 0
    finally:
        m.destroy()


def test_cap_below_one_layer_steps_working_set_is_a_clean_create_error(P):
    wl = synth.WORKLOADS["tiny_fp32"]
    for max_batch, cap in ((1, 1), (4, 7)):  # working sets min(E, k * max_batch) = 2 and 8
        cfg = P.make_config(wl.d, wl.n_experts, wl.top_k, wl.d_ff, wl.n_layers, wl.wdtype, wl.adtype, cap_slots=cap,
                            max_batch=max_batch)
        with pytest.raises(P.MoEError) as ei:
            P.MoE(cfg)
        assert ei.value.status == ERR["capacity"]


def test_pool_larger_than_the_device_is_a_clean_create_error(P):
    # 64 x 256 experts of 50 MB (d = 4096, d_ff = 2048) with a 2 TB cap: 824 GB of device pool; its
    # allocation (the first one moe_create makes) fails at once
    cfg = P.make_config(4096, 256, 8, 2048, 64, "bf16", "bf16", cap_bytes=2 * 10 ** 12)
    with pytest.raises(P.MoEError) as ei:
        P.MoE(cfg)
    assert ei.value.status == ERR["oom"]
