"""The allocation-free routing entry point (moe_route_noalloc), through the C ABI.

moe_route_noalloc serves callers that cannot allocate device memory when they route (a runtime
that reserves all device memory up front, a plug-in inside a host process that owns the
allocator): its logits go to a fixed scratch array inside the library. This file is collected
last so that a run stopping at its first failure has already run every other test.

GPU checks, each on two calls in a row (the scratch keeps the previous call's contents) and on
one call with every token as a row:
  - ids and gates are bit-identical to the routing moe_decode_step computes on the same inputs
    (the two share the logit arithmetic and the top-k code);
  - ids equal the fp64 oracle's except where the oracle's k-th and (k+1)-th logits lie within the
    near-tie margin, gates within the fp32 tolerance;
  - a router row of NaNs still yields expert ids inside [0, E).
Cases: bf16 at the layer's full size, fp32 (E = 8), renorm off, E = 250 and E = 256 (not
multiples of the 32-lane stride, and the largest E), 64 rows (the largest batch).
CPU checks: sizes beyond the scratch and misaligned pointers are rejected before any launch.
"""
import ctypes

import numpy as np
import pytest

import oracle
import synth
from tests.gpu_harness import check_routing

# (workload, tokens, renorm): tokens are also the row count of the batched call
CASES = {
    "layer_bf16": (synth.WORKLOADS["layer_bf16"].replace(n_layers=2, tokens=4, cap_slots=16), True),
    "tiny_fp32": (synth.WORKLOADS["tiny_fp32"].replace(tokens=6), True),
    "e250_raw_softmax": (synth.Workload("e250", d=256, n_experts=250, top_k=8, d_ff=128, n_layers=1, wdtype="bf16",
                                        adtype="bf16", tokens=5, batch=1, rho=0.8, cap_slots=250), False),
    "e256_k16_64rows": (synth.Workload("e256", d=384, n_experts=256, top_k=16, d_ff=64, n_layers=1, wdtype="bf16",
                                       adtype="bf16", tokens=64, batch=1, rho=0.8, cap_slots=256), True),
}


def _device_inputs(wl):
    import torch

    dev = torch.device("cuda", 0)
    hidden = synth.hidden_all(wl)  # [T x L x 1 x d]
    if wl.adtype == "fp32":
        hid = torch.from_numpy(hidden).to(dev)
        routers = [torch.from_numpy(synth.router_weights(wl, l)).to(dev) for l in range(wl.n_layers)]
    else:
        hid = torch.from_numpy(hidden.view(np.int16)).to(dev).view(torch.bfloat16)
        routers = [torch.from_numpy(synth.router_weights(wl, l).view(np.int16)).to(dev).view(torch.bfloat16)
                   for l in range(wl.n_layers)]
    return hidden, hid, routers


def _noalloc_all(P, wl, hid, routers, renorm):
    """Per (t, l): two single-row calls in a row (both kept), then one call over all T rows."""
    import torch

    T, L = wl.tokens, wl.n_layers
    single = [np.empty((T, L, wl.top_k), np.int32), np.empty((T, L, wl.top_k), np.float32)]
    twice = [np.empty_like(single[0]), np.empty_like(single[1])]
    for t in range(T):
        for l in range(L):
            for dst in (single, twice):
                idx, gate = P.route_noalloc(routers[l], hid[t, l].contiguous(), wl.top_k, renorm=renorm)
                torch.cuda.synchronize()
                dst[0][t, l], dst[1][t, l] = idx.cpu().numpy()[0], gate.cpu().numpy()[0]
    rows = [np.empty_like(single[0]), np.empty_like(single[1])]
    for l in range(L):
        idx, gate = P.route_noalloc(routers[l], hid[:, l, 0].contiguous(), wl.top_k, renorm=renorm)
        torch.cuda.synchronize()
        rows[0][:, l], rows[1][:, l] = idx.cpu().numpy(), gate.cpu().numpy()
    return single, twice, rows


@pytest.mark.gpu
@pytest.mark.parametrize("case", sorted(CASES))
def test_noalloc_routing_is_the_decode_steps_bit_for_bit(case):
    import torch

    import paper_2605_29135_gb300 as P
    from paper_2605_29135_gb300.workload import create_for_workload

    P.build()
    wl, renorm = CASES[case]
    _, hid, routers = _device_inputs(wl)
    m = create_for_workload(wl, renorm=renorm)
    try:
        out = torch.empty_like(hid[0])
        ref_idx = np.empty((wl.tokens, wl.n_layers, wl.top_k), np.int32)
        ref_gate = np.empty(ref_idx.shape, np.float32)
        for t in range(wl.tokens):
            m.decode_step(hid[t], out)
            i, g = m.get_last_routing()
            ref_idx[t], ref_gate[t] = i[:, 0], g[:, 0]
    finally:
        m.destroy()
    torch.cuda.synchronize()
    for name, (idx, gate) in zip(("first call", "second call", "all rows"), _noalloc_all(P, wl, hid, routers, renorm)):
        assert np.array_equal(idx, ref_idx), f"{name}: expert ids differ from the decode step's"
        assert np.array_equal(gate.view(np.uint32), ref_gate.view(np.uint32)), f"{name}: gates differ in some bit"


@pytest.mark.gpu
@pytest.mark.parametrize("case", sorted(CASES))
def test_noalloc_routing_matches_the_oracle(case):
    import paper_2605_29135_gb300 as P

    P.build()
    wl, renorm = CASES[case]
    hidden, hid, routers = _device_inputs(wl)
    T, L, k = wl.tokens, wl.n_layers, wl.top_k
    oidx = np.empty((T, L, k), np.int32)
    ogate = np.empty((T, L, k))
    oz = np.empty((T, L, wl.n_experts))
    for l in range(L):
        W = oracle.widen(wl.router_dtype, synth.router_weights(wl, l), wl.n_experts, wl.d)
        for t in range(T):
            oidx[t, l], ogate[t, l], oz[t, l], _ = oracle.router(W, synth.act_to_f64(hidden[t, l, 0], wl.adtype), k,
                                                                renorm=renorm)
    for name, (idx, gate) in zip(("first call", "second call", "all rows"), _noalloc_all(P, wl, hid, routers, renorm)):
        check_routing(idx, oidx, oz, k)
        same = np.all(idx == oidx, axis=-1)
        assert same.mean() > 0.5, f"{name}: most rows should carry no near-tie flip"
        np.testing.assert_allclose(gate[same], ogate[same], rtol=2e-5, atol=1e-6, err_msg=name)


@pytest.mark.gpu
def test_noalloc_ids_stay_in_range_when_logits_are_nan():
    import torch

    import paper_2605_29135_gb300 as P

    P.build()
    wl = CASES["e250_raw_softmax"][0]
    _, hid, routers = _device_inputs(wl)
    w = routers[0].clone()
    w[3] = float("nan")
    w[77] = -float("nan")
    for renorm in (True, False):
        for _ in range(2):
            idx, _ = P.route_noalloc(w, hid[:, 0, 0].contiguous(), wl.top_k, renorm=renorm)
            torch.cuda.synchronize()
            ids = idx.cpu().numpy()
            assert ids.min() >= 0 and ids.max() < wl.n_experts
            assert all(len(set(r.tolist())) == wl.top_k for r in ids), "an expert was selected twice in a row"


def test_noalloc_rejects_sizes_beyond_the_scratch():
    from paper_2605_29135_gb300 import _lib
    from paper_2605_29135_gb300.buildsys import build

    build()
    lib = _lib.load()
    dummy = ctypes.c_void_p(256)  # never dereferenced: the argument checks run first
    too_many_rows = lib.moe_route_noalloc(dummy, dummy, 65, 128, 2048, 8, 1, 1, dummy, dummy, None)
    too_many_experts = lib.moe_route_noalloc(dummy, dummy, 1, 257, 2048, 8, 1, 1, dummy, dummy, None)
    assert too_many_rows == -4 and too_many_experts == -4  # MOE_ERR_CAPACITY
    assert lib.moe_route_noalloc(dummy, dummy, 1, 128, 2048, 17, 1, 1, dummy, dummy, None) == -1


def test_noalloc_rejects_misaligned_pointers_before_any_launch():
    from paper_2605_29135_gb300 import _lib
    from paper_2605_29135_gb300.buildsys import build

    build()
    lib = _lib.load()
    a, odd = ctypes.c_void_p(256), ctypes.c_void_p(258)  # never dereferenced
    # w_r and hidden are read as 16-byte vectors; idx and gate are 4-byte stores
    assert lib.moe_route_noalloc(odd, a, 1, 128, 2048, 8, 1, 1, a, a, None) == -1
    assert lib.moe_route_noalloc(a, odd, 1, 128, 2048, 8, 1, 1, a, a, None) == -1
    assert lib.moe_route_noalloc(a, a, 1, 128, 2048, 8, 1, 1, odd, a, None) == -1
    assert lib.moe_route_noalloc(a, a, 1, 128, 2048, 8, 1, 1, a, odd, None) == -1
