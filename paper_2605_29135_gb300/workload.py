"""Load a seeded synthetic workload (``synth``) into a library handle.

Router weights go to the device; every expert is generated and registered into the pinned
host tier in parallel (the ctypes calls release the GIL, so generation and repacking run on
all host cores).
"""
from __future__ import annotations

import os
import threading
from concurrent.futures import ThreadPoolExecutor

import numpy as np

from . import MoE, make_config


def config_for(wl, cap_slots=None, device=0, trace_capacity=1 << 22, renorm=True, schedule="device", miss_ctas=0,
               batched_path="auto", policy="lru", lookahead=False):
    return make_config(wl.d, wl.n_experts, wl.top_k, wl.d_ff, wl.n_layers, wl.wdtype, wl.adtype,
                       cap_slots=wl.cap_slots if cap_slots is None else cap_slots, renorm=renorm, device=device,
                       max_batch=wl.batch, trace_capacity=trace_capacity, schedule=schedule, miss_ctas=miss_ctas,
                       batched_path=batched_path, policy=policy, lookahead=lookahead)


def create_for_workload(wl, cap_slots=None, device=0, trace_capacity=1 << 22, threads=None,
                        schedule="device", miss_ctas=0, batched_path="auto", renorm=True, policy="lru",
                        lookahead=False) -> MoE:
    import synth

    m = MoE(config_for(wl, cap_slots, device, trace_capacity, renorm=renorm, schedule=schedule, miss_ctas=miss_ctas,
                       batched_path=batched_path, policy=policy, lookahead=lookahead))
    try:
        for layer in range(wl.n_layers):
            m.set_router(layer, synth.router_weights(wl, layer))
        local = threading.local()

        def one(job):
            layer, e = job
            tmp = getattr(local, "tmp", None)
            if tmp is None:
                tmp = local.tmp = np.empty(wl.d * wl.d_ff, dtype=np.float32)
            w = synth.expert_weights(wl, layer, e, tmp)
            m.register_host_experts(layer, e, w.gate, w.up, w.down, w.scales_flat())

        jobs = [(layer, e) for layer in range(wl.n_layers) for e in range(wl.n_experts)]
        with ThreadPoolExecutor(max_workers=threads or os.cpu_count()) as ex:
            for _ in ex.map(one, jobs):
                pass
    except BaseException:
        m.destroy()
        raise
    return m


def create_decoder_for_workload(dw, cap_slots=None, max_tokens=None, device=0, trace_capacity=1 << 22,
                                threads=None):
    """A MoE handle for dw.moe (device schedule, batch 1) and a chained decoder around it, loaded
    with dw's seeded attention weights and KV-cache prefix (dw.ctx positions per layer), with room
    for max_tokens decode tokens (default: dw.moe.tokens). Returns (moe, decoder)."""
    import synth

    from . import Decoder

    m = create_for_workload(dw.moe, cap_slots=cap_slots, device=device, trace_capacity=trace_capacity,
                            threads=threads)
    try:
        T = dw.moe.tokens if max_tokens is None else max_tokens
        dec = Decoder(m, dw.n_heads, dw.n_kv_heads, dw.head_dim, max_pos=dw.ctx + T, eps=dw.eps,
                      rope_theta=dw.rope_theta)
        try:
            for layer in range(dw.moe.n_layers):
                a = synth.attention_weights(dw, layer)
                dec.set_layer(layer, a["wq"], a["wk"], a["wv"], a["wo"], a["norm_in"], a["norm_post"], a["norm_q"],
                              a["norm_k"])
                K, V = synth.kv_prefix(dw, layer)
                dec.set_cache(layer, K, V)
        except BaseException:
            dec.destroy()
            raise
    except BaseException:
        m.destroy()
        raise
    return m, dec
