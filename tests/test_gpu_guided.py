"""Router-guided replacement (MOE_POLICY_GUIDED, device schedule, batch 1 and batched) through the C
ABI against the oracle's guided step.

The device ranks experts by its fp32 logits (moe_get_last_logits). Those ranks must agree with the
oracle's fp64 logits up to swaps of experts whose oracle logits lie within the near-tie bound. The
oracle replayed with the device's selections and ranks must then give the device's residency trace
bit for bit. Outputs are within the dtype's tolerance of the fp64 oracle and bit-identical to the
LRU policy's (the policy only changes where the weights are read from)."""
import numpy as np
import pytest

import oracle
import synth
from tests.gpu_harness import NEAR_TIE, TOL, rel_l2_rows, trace_tuples

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def P():
    import paper_2605_29135_gb300 as P

    P.build()
    return P


def _run(wl, cap, policy, preload=False, batched_path="auto", schedule="device"):
    """Decode every token on the device; returns hidden, outputs, selections, logits, trace, stats."""
    import torch

    from paper_2605_29135_gb300.workload import create_for_workload

    hidden = synth.hidden_all(wl)
    T, B = hidden.shape[0], hidden.shape[2]
    dev = torch.device("cuda", 0)
    fp32 = wl.adtype == "fp32"
    hid = torch.from_numpy(hidden.view(np.float32) if fp32 else hidden.view(np.int16)).to(dev)
    if not fp32:
        hid = hid.view(torch.bfloat16)
    out = torch.empty(hid.shape, dtype=hid.dtype, device=dev)
    idx = np.empty((T, wl.n_layers, B, wl.top_k), dtype=np.int32)
    z = np.empty((T, wl.n_layers, B, wl.n_experts), dtype=np.float32)
    m = create_for_workload(wl, cap_slots=cap, schedule=schedule, policy=policy, batched_path=batched_path)
    try:
        if preload:
            m.preload()
        for t in range(T):
            m.decode_step(hid[t], out[t], batch=B)
            i, _ = m.get_last_routing()
            idx[t] = i[:, :B]
            if policy == "guided":
                z[t] = m.get_last_logits()[:, :B]
        torch.cuda.synchronize()
        tr = m.get_residency_trace()
        stats = m.get_stats()
    finally:
        m.destroy()
    o = out.float().cpu().numpy().astype(np.float64)
    return hidden, o, idx, z, tr, stats


def _device_ranks(z32):
    """Ranks from the device's fp32 logits: descending, ties to the lower id."""
    r = np.empty(z32.shape, dtype=np.int32)
    for pos in np.ndindex(*z32.shape[:-1]):
        order = np.argsort(-z32[pos].astype(np.float64), kind="stable")
        r[pos][order] = np.arange(z32.shape[-1], dtype=np.int32)
    return r


def _check_ranks(ranks, z64, idx):
    """Per sequence: the device's order of a layer-step's experts is the oracle's up to near-ties,
    and its top-k selection is the head of that order."""
    k = idx.shape[-1]
    np.testing.assert_array_equal(idx, np.argsort(ranks, axis=-1)[..., :k])
    for pos in np.ndindex(*ranks.shape[:-1]):
        order = np.argsort(ranks[pos])
        zs = z64[pos][order]
        assert (zs[1:] <= zs[:-1] + NEAR_TIE).all(), f"rank order differs beyond a near-tie at {pos}"


def _replay(wl, cap, hidden, idx, ranks, preload=False, compute_out=True):
    """The oracle with the device's selections and, per layer-step, its best rank over the batch."""
    orc = oracle.Oracle.for_workload(wl, cap_slots=cap, policy="guided", keep_slot_copies=compute_out)
    if preload:
        orc.preload()
    best = ranks.min(axis=2)  # [T x L x E]
    res = [orc.decode_step(hidden[t], compute_out=compute_out, forced_idx=idx[t], forced_ranks=best[t])
           for t in range(hidden.shape[0])]
    return res


def _oracle_z(wl, hidden):
    # logits only: a pool holding every expert, so any batch's needed set fits
    orc = oracle.Oracle.for_workload(wl, cap_slots=wl.n_gid, keep_slot_copies=False, policy="guided")
    return np.stack([orc.decode_step(hidden[t], compute_out=False).z for t in range(hidden.shape[0])])


SCHEDULES = ["device", "host_copy_engine"]


@pytest.mark.parametrize("schedule", SCHEDULES)
@pytest.mark.parametrize("cap", [2, 3, 5])
def test_tiny_guided_trace_and_outputs(P, cap, schedule):
    wl = synth.WORKLOADS["tiny_fp32"].replace(n_layers=2)
    hidden, out, idx, z, tr, stats = _run(wl, cap, "guided", schedule=schedule)
    ranks = _device_ranks(z)
    _check_ranks(ranks, _oracle_z(wl, hidden), idx)
    res = _replay(wl, cap, hidden, idx, ranks)
    np.testing.assert_array_equal(trace_tuples(tr), trace_tuples(np.concatenate([r.records for r in res])))
    assert rel_l2_rows(out, np.stack([r.out for r in res])).max() <= TOL["fp32"]
    assert stats["misses"] == int((tr["kind"] == 1).sum()) and stats["evictions"] == int((tr["evicted"] >= 0).sum())
    _, out_lru, _, _, tr_lru, _ = _run(wl, cap, "lru", schedule=schedule)
    np.testing.assert_array_equal(out, out_lru)  # same arithmetic whatever the slot contents


@pytest.mark.parametrize("schedule", SCHEDULES)
def test_guided_preload(P, schedule):
    wl = synth.WORKLOADS["tiny_fp32"].replace(n_layers=2, tokens=32)
    hidden, out, idx, z, tr, _ = _run(wl, 6, "guided", preload=True, schedule=schedule)
    res = _replay(wl, 6, hidden, idx, _device_ranks(z), preload=True, compute_out=False)
    np.testing.assert_array_equal(trace_tuples(tr), trace_tuples(np.concatenate([r.records for r in res])))


def test_layer_bf16_guided(P):
    wl = synth.WORKLOADS["layer_bf16"].replace(tokens=256)
    hidden, out, idx, z, tr, _ = _run(wl, wl.cap_slots, "guided")
    ranks = _device_ranks(z)
    _check_ranks(ranks, _oracle_z(wl, hidden), idx)
    res = _replay(wl, wl.cap_slots, hidden, idx, ranks, compute_out=False)
    np.testing.assert_array_equal(trace_tuples(tr), trace_tuples(np.concatenate([r.records for r in res])))
    orc = oracle.Oracle.for_workload(wl, keep_slot_copies=False)
    for t in (0, 100, 255):
        ref, _, _ = orc.moe_layer(0, hidden[t, 0, 0], forced_idx=idx[t, 0, 0])
        assert rel_l2_rows(out[t, 0, 0], ref) <= TOL["bf16"]


@pytest.mark.parametrize("schedule", SCHEDULES)
@pytest.mark.parametrize("name", ["stack48_bf16", "stack48_int4"])
def test_stack48_guided_512_tokens(P, name, schedule):
    wl = synth.WORKLOADS[name].replace(tokens=512)
    hidden, out, idx, z, tr, stats = _run(wl, wl.cap_slots, "guided", schedule=schedule)
    ranks = _device_ranks(z)
    _check_ranks(ranks, _oracle_z(wl, hidden), idx)
    res = _replay(wl, wl.cap_slots, hidden, idx, ranks, compute_out=False)
    np.testing.assert_array_equal(trace_tuples(tr), trace_tuples(np.concatenate([r.records for r in res])))
    orc = oracle.Oracle.for_workload(wl, keep_slot_copies=False)
    for t, l in [(0, 0), (255, 20), (511, 47)]:
        ref, _, _ = orc.moe_layer(l, hidden[t, l, 0], forced_idx=idx[t, l, 0])
        assert rel_l2_rows(out[t, l, 0], ref) <= TOL[wl.wdtype]
    # the point of the policy: fewer misses than LRU on the same tokens
    _, _, _, _, _, stats_lru = _run(wl, wl.cap_slots, "lru", schedule=schedule)
    assert stats["misses"] < stats_lru["misses"]


@pytest.mark.parametrize("path", ["auto", "cuda_cores"])
def test_tiny_batched_guided(P, path):
    # bf16, d = 256, d_ff = 128: "auto" takes the tensor-core kernel, "cuda_cores" the GEMV one
    wl = synth.WORKLOADS["tiny_fp32"].replace(wdtype="bf16", adtype="bf16", n_layers=3, batch=4, tokens=24)
    cap = 8
    hidden, out, idx, z, tr, stats = _run(wl, cap, "guided", batched_path=path)
    ranks = _device_ranks(z)
    _check_ranks(ranks, _oracle_z(wl, hidden), idx)
    res = _replay(wl, cap, hidden, idx, ranks)
    np.testing.assert_array_equal(trace_tuples(tr), trace_tuples(np.concatenate([r.records for r in res])))
    assert rel_l2_rows(out, np.stack([r.out for r in res])).max() <= TOL["bf16"]


def test_batch64_guided_keeps_part_of_the_pool(P):
    # 64 sequences put nearly every expert of a layer at rank 0, so ties to the more recent use
    # decide; unlike LRU, part of the pool then survives from one token to the next
    wl = synth.WORKLOADS["stack48_batch64"].replace(tokens=6)
    hidden, out, idx, z, tr, stats = _run(wl, wl.cap_slots, "guided")
    ranks = _device_ranks(z)
    _check_ranks(ranks, _oracle_z(wl, hidden), idx)
    res = _replay(wl, wl.cap_slots, hidden, idx, ranks, compute_out=False)
    np.testing.assert_array_equal(trace_tuples(tr), trace_tuples(np.concatenate([r.records for r in res])))
    assert stats["hits"] > 0
