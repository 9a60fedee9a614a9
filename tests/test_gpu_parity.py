"""GPU parity: the CUDA path through the C ABI against the fp64 oracle on the same seeded inputs.

Per workload: the residency trace is bit-exact; top-k ids are exact except near-ties (oracle
logit gap < 1e-4 around the k-th); gates agree to fp32 rounding; outputs have relative L2 error
per (token, layer) row <= 1e-5 (fp32), 1e-2 (bf16), 3e-2 (int4, against the oracle on the same
dequantised weights). Sizes span several tiles with ragged tails; the Qwen3-30B-A3B-shaped
workloads run at full size in the configuration bench.py times, with outputs checked on sampled
(token, layer) rows.
"""
import functools
from concurrent.futures import ThreadPoolExecutor

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


# "host_lookahead": the host copy-engine schedule routing layer l + 1 while layer l computes; it
# must give the same trace and outputs as the others
SCHEDULES = ["device", "host_copy_engine", "host_lookahead"]
_ORACLE_CACHE = {}


def _create(wl, cap, schedule="device"):
    from paper_2605_29135_gb300.workload import create_for_workload

    if schedule == "host_lookahead":
        return create_for_workload(wl, cap_slots=cap, schedule="host_copy_engine", lookahead=True)
    if schedule == "device_lookahead":
        return create_for_workload(wl, cap_slots=cap, schedule="device", lookahead=True)
    return create_for_workload(wl, cap_slots=cap, schedule=schedule)


def _oracle_routing(wl, cap, tokens, hidden, routers):
    key = (wl, cap, tokens)
    if key not in _ORACLE_CACHE:
        _ORACLE_CACHE.clear()
        _ORACLE_CACHE[key] = oracle_trace(wl, hidden, cap, routers=routers)
    return _ORACLE_CACHE[key]


def _parity(P, wl, cap, tokens, samples=None, threads=8, schedule="device"):
    hidden = synth.hidden_all(wl, tokens)
    m = _create(wl, cap, schedule)
    try:
        out, idx, gate = run_gpu(m, hidden, wl.adtype)
        tr = m.get_residency_trace()
        stats = m.get_stats()
    finally:
        m.destroy()
    routers = [synth.router_weights(wl, l) for l in range(wl.n_layers)]
    oidx, oz, otr = _oracle_routing(wl, cap, tokens, hidden, routers)
    flips = check_routing(idx, oidx, oz, wl.top_k)
    if flips:
        _, _, otr = oracle_trace(wl, hidden, cap, forced_idx=idx, routers=routers)
    np.testing.assert_array_equal(trace_tuples(tr), trace_tuples(otr))
    assert stats["hits"] + stats["misses"] == len(tr)
    assert stats["misses"] == int((tr["kind"] == 1).sum())
    assert stats["evictions"] == int((tr["evicted"] >= 0).sum())
    # outputs on sampled rows (all rows when samples is None), layer by layer so that the rows of
    # one layer share the generated experts they route to
    orc = oracle.Oracle.for_workload(wl, keep_slot_copies=False, routers=routers,
                                     experts=functools.lru_cache(maxsize=512)(
                                         lambda l, e: synth.expert_weights(wl, l, e)))
    if samples is None:
        samples = [(t, l) for t in range(tokens) for l in range(wl.n_layers)]
    samples = sorted(samples, key=lambda tl: (tl[1], tl[0]))

    def one(tl):
        t, l = tl
        ref, _, g = orc.moe_layer(l, hidden[t, l, 0], forced_idx=idx[t, l, 0])
        return t, l, ref, g

    with ThreadPoolExecutor(max_workers=threads) as ex:
        res = list(ex.map(one, samples))
    errs = []
    for t, l, ref, g in res:
        np.testing.assert_allclose(gate[t, l, 0], g, rtol=2e-5, atol=1e-6)
        errs.append(rel_l2_rows(out[t, l, 0], ref))
    errs = np.array(errs)
    assert errs.max() <= TOL[wl.wdtype], f"max rel L2 {errs.max():.3e} (mean {errs.mean():.3e})"
    return out, tr, errs, flips


@pytest.mark.parametrize("schedule", SCHEDULES)
def test_tiny_fp32_full_run(P, schedule):
    wl = synth.WORKLOADS["tiny_fp32"]
    out, tr, errs, _ = _parity(P, wl, wl.cap_slots, wl.tokens, schedule=schedule)
    assert (tr["kind"] == 0).sum() > 0 and (tr["evicted"] >= 0).sum() > 0


@pytest.mark.parametrize("name", ["tiny_fp32", "layer_bf16"])
def test_cap_invariance_bit_exact_across_schedules(P, name):
    # outputs do not depend on the cap (residency only changes where weights are read from) nor
    # on the schedule: the same kernels' arithmetic runs on slot or host-tier bytes
    wl = synth.WORKLOADS[name]
    tokens = min(wl.tokens, 96)
    hidden = synth.hidden_all(wl, tokens)
    outs = []
    for cap, schedule in ((wl.cap_slots, "device"), (wl.n_gid, "device"), (wl.cap_slots, "host_copy_engine"),
                          (wl.cap_slots, "host_lookahead")):
        m = _create(wl, cap, schedule)
        try:
            outs.append(run_gpu(m, hidden, wl.adtype)[0])
        finally:
            m.destroy()
    np.testing.assert_array_equal(outs[0], outs[1])
    np.testing.assert_array_equal(outs[0], outs[2])
    np.testing.assert_array_equal(outs[0], outs[3])


RAGGED = {
    "fp32": synth.Workload("ragged_fp32", d=100, n_experts=5, top_k=2, d_ff=36, n_layers=2, wdtype="fp32",
                           adtype="fp32", tokens=24, batch=1, rho=0.9, cap_slots=3),
    "bf16": synth.Workload("ragged_bf16", d=640, n_experts=24, top_k=5, d_ff=200, n_layers=3, wdtype="bf16",
                           adtype="bf16", tokens=24, batch=1, rho=0.8, cap_slots=7),
    "int4": synth.Workload("ragged_int4", d=384, n_experts=12, top_k=3, d_ff=256, n_layers=2, wdtype="int4",
                           adtype="bf16", tokens=24, batch=1, rho=0.8, cap_slots=4),
    "bf16_wide": synth.Workload("wide_bf16", d=4096, n_experts=256, top_k=16, d_ff=1536, n_layers=1,
                                wdtype="bf16", adtype="bf16", tokens=6, batch=1, rho=0.8, cap_slots=20),
}


@pytest.mark.parametrize("schedule", SCHEDULES)
@pytest.mark.parametrize("name", list(RAGGED))
def test_ragged_shapes(P, name, schedule):
    wl = RAGGED[name]
    _parity(P, wl, wl.cap_slots, wl.tokens, schedule=schedule)


@pytest.mark.parametrize("schedule", SCHEDULES)
def test_layer_bf16_full_2048_tokens(P, schedule):
    wl = synth.WORKLOADS["layer_bf16"]
    samples = [(t, 0) for t in range(0, wl.tokens, 64)] + [(wl.tokens - 1, 0)]
    _parity(P, wl, wl.cap_slots, wl.tokens, samples=samples, schedule=schedule)


@pytest.mark.parametrize("schedule", SCHEDULES)
@pytest.mark.parametrize("name", ["stack48_int4", "stack48_bf16"])
def test_stack48_full_2048_tokens(P, name, schedule):
    # the benchmarked configurations: every residency record of the 2048 tokens; outputs of every
    # 64th token (and the last) in all 48 layers on the device schedule the bench times, of 24
    # (token, layer) rows on the others
    wl = synth.WORKLOADS[name]
    if schedule == "device":
        samples = [(t, l) for t in list(range(0, wl.tokens, 64)) + [wl.tokens - 1] for l in range(wl.n_layers)]
    else:
        samples = [(t, l) for t in (0, 1023, 2047) for l in range(0, 48, 6)]
    _, tr, errs, flips = _parity(P, wl, wl.cap_slots, wl.tokens, samples=samples, threads=16, schedule=schedule)
    assert len(tr) == wl.tokens * wl.n_layers * wl.top_k


@pytest.mark.parametrize("schedule", SCHEDULES)
@pytest.mark.parametrize("cap", [4, 8])
def test_preload_then_decode_matches_oracle(P, schedule, cap):
    wl = synth.WORKLOADS["tiny_fp32"]
    hidden = synth.hidden_all(wl)
    m = _create(wl, cap, schedule)
    try:
        assert m.preload() == min(cap, wl.n_gid)
        out, idx, _ = run_gpu(m, hidden, wl.adtype)
        tr = m.get_residency_trace()
    finally:
        m.destroy()
    orc = oracle.Oracle.for_workload(wl, cap_slots=cap)
    orc.preload()
    recs, ref = [], []
    for t in range(wl.tokens):
        r = orc.decode_step(hidden[t], forced_idx=idx[t])
        recs.append(r.records)
        ref.append(r.out)
    np.testing.assert_array_equal(trace_tuples(tr), trace_tuples(np.concatenate(recs)))
    assert rel_l2_rows(out, np.stack(ref)).max() <= TOL["fp32"]
    if cap >= wl.n_gid:
        assert (tr["kind"] == 0).all()


# The device schedule with exact layer lookahead: one kernel routes every layer, CTA 0 then decides
# the layers' lookups in order ahead of the compute (cap >= 2 * top_k, or every expert resident).
# Same trace and outputs as the layer-by-layer kernel, bit for bit. The workers take layers in
# groups of P = 2 from 4 * top_k slots (else 1) and run skewed (a group's down rows after the next
# group's gate/up rows) from 3 * P * top_k slots or with every expert resident. tiny_fp32 has
# top_k = 2: 8 layers at cap 6 run P = 1 skewed, cap 11 P = 2 unskewed, cap 12 P = 2 skewed.
LOOKAHEAD = {
    "tiny3_fp32_cap4": synth.WORKLOADS["tiny_fp32"].replace(n_layers=3, cap_slots=4),
    "tiny3_fp32_cap8": synth.WORKLOADS["tiny_fp32"].replace(n_layers=3, cap_slots=8),
    "tiny8_fp32_cap6_p1_skewed": synth.WORKLOADS["tiny_fp32"].replace(n_layers=8, tokens=32, cap_slots=6),
    "tiny8_fp32_cap11_p2": synth.WORKLOADS["tiny_fp32"].replace(n_layers=8, tokens=32, cap_slots=11),
    "tiny8_fp32_cap12_p2_skewed": synth.WORKLOADS["tiny_fp32"].replace(n_layers=8, tokens=32, cap_slots=12),
    "tiny8_bf16_cap12_p2_skewed": synth.WORKLOADS["tiny_fp32"].replace(n_layers=8, tokens=32, cap_slots=12,
                                                                       wdtype="bf16", adtype="bf16"),
    "ragged_fp32": RAGGED["fp32"].replace(cap_slots=4),
    "ragged_bf16": RAGGED["bf16"].replace(cap_slots=10),
    "ragged_int4": RAGGED["int4"].replace(cap_slots=6),
    "tiny3_fp32_resident": synth.WORKLOADS["tiny_fp32"].replace(n_layers=3, cap_slots=24),
}


@pytest.mark.parametrize("name", list(LOOKAHEAD))
def test_device_lookahead_matches_oracle_and_the_layer_by_layer_kernel(P, name):
    wl = LOOKAHEAD[name]
    out, tr, _, _ = _parity(P, wl, wl.cap_slots, wl.tokens, schedule="device_lookahead")
    if wl.cap_slots < wl.n_gid:
        assert (tr["evicted"] >= 0).sum() > 0
    out2, tr2, _, _ = _parity(P, wl, wl.cap_slots, wl.tokens, schedule="device")
    np.testing.assert_array_equal(out, out2)
    np.testing.assert_array_equal(trace_tuples(tr), trace_tuples(tr2))


@pytest.mark.parametrize("name", ["stack48_int4", "stack48_bf16"])
def test_device_lookahead_stack48_2048_tokens(P, name):
    wl = synth.WORKLOADS[name]
    samples = [(t, l) for t in (0, 1023, 2047) for l in range(0, 48, 6)]
    _, tr, _, _ = _parity(P, wl, wl.cap_slots, wl.tokens, samples=samples, threads=16, schedule="device_lookahead")
    assert len(tr) == wl.tokens * wl.n_layers * wl.top_k


def test_device_lookahead_preload_and_small_caps(P):
    wl = LOOKAHEAD["tiny3_fp32_cap8"]
    hidden = synth.hidden_all(wl)
    m = _create(wl, 10, "device_lookahead")
    try:
        assert m.preload() == 10
        out, idx, _ = run_gpu(m, hidden, wl.adtype)
        tr = m.get_residency_trace()
    finally:
        m.destroy()
    orc = oracle.Oracle.for_workload(wl, cap_slots=10)
    orc.preload()
    recs = [orc.decode_step(hidden[t], compute_out=False, forced_idx=idx[t]).records for t in range(wl.tokens)]
    np.testing.assert_array_equal(trace_tuples(tr), trace_tuples(np.concatenate(recs)))
    with pytest.raises(P.MoEError) as ei:
        _create(wl, 3, "device_lookahead")  # below 2 * top_k = 4 slots
    assert ei.value.status == -1 and "slots" in str(ei.value)
