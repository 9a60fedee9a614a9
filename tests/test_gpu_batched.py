"""GPU parity of the batched decode step (max_batch > 1) against the fp64 oracle.

Per layer-step the needed experts are the union of all sequences' top-k choices; the oracle
runs one lookup-table step for that union (one record per distinct expert, ascending id) and
evaluates every sequence's experts. Checks, through the C ABI, on the same seeded inputs:
the residency trace bit-exact; top-k ids exact except near-ties; gates to fp32 rounding;
outputs per (token, layer, sequence) row within the dtype's relative L2 bound. Shapes span
several work items with ragged tails (d, d_ff not multiples of the item sizes, odd batch
sizes), a Qwen3-30B-A3B-shaped layer at batch 64, and the 48-layer stack at batch 64 with
a 6 GB pool cap (635 slots) for a few steps. bf16 shapes whose d is a multiple of 128 and d_ff
of 64 run both expert-FFN paths: tensor cores (tcgen05 grouped GEMM, pairs per expert padded
to 16, 32, 48 or 64 columns) and CUDA cores.
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


def _create(wl, cap, **kw):
    from paper_2605_29135_gb300.workload import create_for_workload

    return create_for_workload(wl, cap_slots=cap, **kw)


def _check_outputs(wl, hidden, idx, gate, out, samples, threads=8):
    routers = [synth.router_weights(wl, l) for l in range(wl.n_layers)]
    # rows in layer order, so that the rows of one layer share the generated experts they route to
    orc = oracle.Oracle.for_workload(wl, keep_slot_copies=False, routers=routers,
                                     experts=functools.lru_cache(maxsize=512)(
                                         lambda l, e: synth.expert_weights(wl, l, e)))
    samples = sorted(samples, key=lambda tlb: (tlb[1], tlb[0], tlb[2]))

    def one(tlb):
        t, l, b = tlb
        ref, _, g = orc.moe_layer(l, hidden[t, l, b], forced_idx=idx[t, l, b])
        return t, l, b, ref, g

    with ThreadPoolExecutor(max_workers=threads) as ex:
        res = list(ex.map(one, samples))
    errs = []
    for t, l, b, ref, g in res:
        np.testing.assert_allclose(gate[t, l, b], g, rtol=2e-5, atol=1e-6)
        errs.append(rel_l2_rows(out[t, l, b], ref))
    errs = np.array(errs)
    assert errs.max() <= TOL[wl.wdtype], f"max rel L2 {errs.max():.3e} (mean {errs.mean():.3e})"
    return errs


def _parity(wl, cap, samples=None, threads=8, preload=False, path="auto"):
    hidden = synth.hidden_all(wl)
    m = _create(wl, cap, batched_path=path)
    try:
        if preload:
            m.preload()
        out, idx, gate = run_gpu(m, hidden, wl.adtype)
        tr = m.get_residency_trace()
        stats = m.get_stats()
    finally:
        m.destroy()
    routers = [synth.router_weights(wl, l) for l in range(wl.n_layers)]
    if preload:
        orc = oracle.Oracle.for_workload(wl, cap_slots=cap, keep_slot_copies=False, routers=routers)
        orc.preload()
        otr = np.concatenate([orc.decode_step(hidden[t], compute_out=False, forced_idx=idx[t]).records
                              for t in range(wl.tokens)])
    else:
        oidx, oz, otr = oracle_trace(wl, hidden, cap, routers=routers)
        if check_routing(idx, oidx, oz, wl.top_k):
            _, _, otr = oracle_trace(wl, hidden, cap, forced_idx=idx, routers=routers)
    np.testing.assert_array_equal(trace_tuples(tr), trace_tuples(otr))
    assert stats["hits"] + stats["misses"] == len(tr)
    assert stats["misses"] == int((tr["kind"] == 1).sum())
    assert stats["evictions"] == int((tr["evicted"] >= 0).sum())
    if samples is None:
        samples = [(t, l, b) for t in range(wl.tokens) for l in range(wl.n_layers) for b in range(wl.batch)]
    _check_outputs(wl, hidden, idx, gate, out, samples, threads)
    return out, tr


BATCHED = {
    "fp32": synth.Workload("b_fp32", d=256, n_experts=8, top_k=2, d_ff=128, n_layers=3, wdtype="fp32",
                           adtype="fp32", tokens=24, batch=4, rho=0.9, cap_slots=13),
    "fp32_ragged": synth.Workload("b_fp32_ragged", d=100, n_experts=5, top_k=2, d_ff=36, n_layers=2, wdtype="fp32",
                                  adtype="fp32", tokens=16, batch=3, rho=0.9, cap_slots=6),
    "bf16_ragged": synth.Workload("b_bf16_ragged", d=640, n_experts=24, top_k=5, d_ff=200, n_layers=3,
                                  wdtype="bf16", adtype="bf16", tokens=10, batch=5, rho=0.8, cap_slots=40),
    "int4": synth.Workload("b_int4", d=384, n_experts=12, top_k=3, d_ff=256, n_layers=2, wdtype="int4",
                           adtype="bf16", tokens=10, batch=6, rho=0.8, cap_slots=14),
    "bf16_wide": synth.Workload("b_bf16_wide", d=4096, n_experts=64, top_k=16, d_ff=1536, n_layers=2,
                                wdtype="bf16", adtype="bf16", tokens=3, batch=7, rho=0.8, cap_slots=80),
    # tensor-core shapes: 3 row tiles of W_d, 3 of [gate; up]; 66 pairs over 20 experts
    "bf16_tc": synth.Workload("b_bf16_tc", d=384, n_experts=20, top_k=6, d_ff=192, n_layers=2, wdtype="bf16",
                              adtype="bf16", tokens=8, batch=11, rho=0.8, cap_slots=28),
    # 128 pairs over 3 experts: 36..46 pairs per expert (N = 48)
    "bf16_dense": synth.Workload("b_bf16_dense", d=256, n_experts=3, top_k=2, d_ff=128, n_layers=3, wdtype="bf16",
                                 adtype="bf16", tokens=6, batch=64, rho=0.8, cap_slots=7),
    # every sequence routes to both experts: 64 pairs per expert (N = 64); the layers' 6 experts
    # cycle through 4 slots, so every request misses and evicts
    "bf16_full": synth.Workload("b_bf16_full", d=256, n_experts=2, top_k=2, d_ff=128, n_layers=3, wdtype="bf16",
                                adtype="bf16", tokens=4, batch=64, rho=0.8, cap_slots=4),
}
TC_SHAPES = ["bf16_wide", "bf16_tc", "bf16_dense", "bf16_full"]


@pytest.mark.parametrize("name", list(BATCHED))
def test_batched_small_shapes(P, name):
    wl = BATCHED[name]
    out, tr = _parity(wl, wl.cap_slots)
    assert (tr["evicted"] >= 0).any()
    assert (tr["kind"] == 0).any() or name == "bf16_full"


@pytest.mark.parametrize("name", TC_SHAPES)
def test_batched_cuda_core_path_on_tensor_core_shapes(P, name):
    wl = BATCHED[name]
    _parity(wl, wl.cap_slots, path="cuda_cores")


@pytest.mark.parametrize("name,path", [("bf16_ragged", "auto"), ("bf16_tc", "auto"), ("bf16_dense", "auto"),
                                       ("bf16_tc", "cuda_cores")])
def test_batched_cap_invariance_bit_exact(P, name, path):
    # residency only changes where the weights are read from: outputs with a capped pool that
    # evicts every step and with every expert resident are identical
    wl = BATCHED[name]
    hidden = synth.hidden_all(wl)
    outs = []
    for cap in (wl.cap_slots, wl.n_gid):
        m = _create(wl, cap, batched_path=path)
        try:
            outs.append(run_gpu(m, hidden, wl.adtype)[0])
        finally:
            m.destroy()
    np.testing.assert_array_equal(outs[0], outs[1])


def test_batched_preload_all_resident_only_hits(P):
    wl = BATCHED["int4"]
    _, tr = _parity(wl, wl.n_gid, preload=True)
    assert (tr["kind"] == 0).all()


def test_batch_size_varies_between_steps(P):
    # a handle made for up to 6 sequences decodes steps of 6, 1, 4 and 6 sequences; the oracle
    # runs the same steps on the same rows
    import torch

    wl = BATCHED["int4"]
    hidden = synth.hidden_all(wl)
    sizes = [6, 1, 4, 6]
    m = _create(wl, wl.cap_slots)
    dev = torch.device("cuda", 0)
    outs, idxs = [], []
    try:
        for t, B in enumerate(sizes):
            h = torch.from_numpy(np.ascontiguousarray(hidden[t, :, :B]).view(np.int16)).to(dev).view(torch.bfloat16)
            o = torch.empty_like(h)
            m.decode_step(h, o, batch=B)
            i, _ = m.get_last_routing()
            idxs.append(i[:, :B].copy())
            outs.append(o.float().cpu().numpy().astype(np.float64))
        tr = m.get_residency_trace()
    finally:
        m.destroy()
    orc = oracle.Oracle.for_workload(wl, keep_slot_copies=False)
    recs = []
    for t, B in enumerate(sizes):
        r = orc.decode_step(np.ascontiguousarray(hidden[t, :, :B]), forced_idx=idxs[t])
        recs.append(r.records)
        assert rel_l2_rows(outs[t], r.out).max() <= TOL[wl.wdtype]
    np.testing.assert_array_equal(trace_tuples(tr), trace_tuples(np.concatenate(recs)))


def test_batch_above_max_is_rejected(P):
    import torch

    wl = BATCHED["fp32"]
    m = _create(wl, wl.cap_slots)
    try:
        h = torch.zeros((wl.n_layers, wl.batch + 1, wl.d), dtype=torch.float32, device="cuda")
        with pytest.raises(P.MoEError) as ei:
            m.decode_step(h, torch.empty_like(h), batch=wl.batch + 1)
        assert ei.value.status == -1  # MOE_ERR_INVALID
    finally:
        m.destroy()


@pytest.mark.parametrize("path", ["auto", "cuda_cores"])
def test_layer_bf16_batch64(P, path):
    # Qwen3-30B-A3B-shaped layers, 64 sequences: 512 routed pairs per layer-step over ~126 experts
    wl = synth.WORKLOADS["layer_bf16"].replace(name="layer_bf16_b64", n_layers=2, batch=64, tokens=4, cap_slots=200)
    rng = np.random.default_rng(0)
    samples = [(t, l, int(b)) for t in range(wl.tokens) for l in range(wl.n_layers)
               for b in rng.choice(64, size=4, replace=False)]
    _parity(wl, wl.cap_slots, samples=samples, threads=16, path=path)


def test_stack48_batch64_all_resident(P):
    # the benchmarked uncapped batch-64 configuration: all 6144 experts preloaded into a 58 GB pool,
    # 48 layers, 64 sequences, tensor-core expert FFN; every request hits
    wl = synth.WORKLOADS["stack48_batch64"].replace(tokens=3, cap_slots=6144)
    samples = [(t, l, b) for t in (0, 2) for l in range(wl.n_layers) for b in (0, 31, 63)]
    _, tr = _parity(wl, wl.cap_slots, samples=samples, threads=16, preload=True)
    assert (tr["kind"] == 0).all() and len(tr) > 0


def test_stack48_batch64_capped_steps(P):
    # the 48-layer bf16 stack at batch 64 under the 6 GB pool cap (635 slots): a few full steps
    wl = synth.WORKLOADS["stack48_batch64"].replace(tokens=3)
    samples = [(t, l, b) for t in (0, 2) for l in (0, 17, 47) for b in (0, 31, 63)]
    _, tr = _parity(wl, wl.cap_slots, samples=samples, threads=16)
    assert (tr["evicted"] >= 0).any()
