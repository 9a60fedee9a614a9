"""The allocation-free routing entry point (moe_route_noalloc) against moe_decode_step's routing.

moe_route_noalloc serves callers that cannot allocate device memory when they route (a runtime
that reserves all device memory up front, a plug-in inside a host process that owns the
allocator): its logits go to a fixed scratch array inside the library. This file is collected
last so that a run stopping at its first failure has already run every other test.

Checks, through the C ABI: two calls in a row (the scratch keeps the previous call's contents)
give the same expert ids as the decode step's router and gates within the fp32 tolerance the
parity tests use; several rows in one call; oversized requests are rejected up front.
"""
import ctypes

import numpy as np
import pytest

import synth


@pytest.mark.gpu
def test_noalloc_routing_matches_decode_step_on_two_calls_in_a_row():
    import torch

    import paper_2605_29135_gb300 as P
    from paper_2605_29135_gb300.buildsys import build
    from paper_2605_29135_gb300.workload import create_for_workload

    build()
    wl = synth.WORKLOADS["layer_bf16"].replace(n_layers=2, tokens=4)
    hidden = synth.hidden_all(wl)  # [T x L x 1 x d] bf16 bits
    dev = torch.device("cuda", 0)
    hid = torch.from_numpy(hidden.view(np.int16)).to(dev).view(torch.bfloat16)
    routers = [torch.from_numpy(synth.router_weights(wl, l).view(np.int16)).to(dev).view(torch.bfloat16)
               for l in range(wl.n_layers)]
    m = create_for_workload(wl)
    try:
        out = torch.empty_like(hid[0])
        ref_idx, ref_gate = [], []
        for t in range(wl.tokens):
            m.decode_step(hid[t], out)
            i, g = m.get_last_routing()
            ref_idx.append(i[:, 0])
            ref_gate.append(g[:, 0])
    finally:
        m.destroy()
    torch.cuda.synchronize()
    # two single-row calls in a row per layer, then one call with every token as a row
    for t in (0, 1):
        for l in range(wl.n_layers):
            idx, gate = P.route_noalloc(routers[l], hid[t, l].contiguous(), wl.top_k)
            torch.cuda.synchronize()
            assert idx.cpu().numpy()[0].tolist() == ref_idx[t][l].tolist()
            np.testing.assert_allclose(gate.cpu().numpy()[0], ref_gate[t][l], rtol=2e-5, atol=1e-6)
    for l in range(wl.n_layers):
        rows = hid[:, l, 0].contiguous()  # [T x d]
        idx, gate = P.route_noalloc(routers[l], rows, wl.top_k)
        torch.cuda.synchronize()
        for t in range(wl.tokens):
            assert idx.cpu().numpy()[t].tolist() == ref_idx[t][l].tolist()
            np.testing.assert_allclose(gate.cpu().numpy()[t], ref_gate[t][l], rtol=2e-5, atol=1e-6)


def test_noalloc_rejects_sizes_beyond_the_scratch():
    from paper_2605_29135_gb300 import _lib
    from paper_2605_29135_gb300.buildsys import build

    build()
    lib = _lib.load()
    dummy = ctypes.c_void_p(16)  # never dereferenced: the size checks run first
    too_many_rows = lib.moe_route_noalloc(dummy, dummy, 65, 128, 2048, 8, 1, 1, dummy, dummy, None)
    too_many_experts = lib.moe_route_noalloc(dummy, dummy, 1, 257, 2048, 8, 1, 1, dummy, dummy, None)
    assert too_many_rows == -4 and too_many_experts == -4  # MOE_ERR_CAPACITY
    assert lib.moe_route_noalloc(dummy, dummy, 1, 128, 2048, 17, 1, 1, dummy, dummy, None) == -1
