"""fp64 oracle of a decode step through a chained stack of decoder blocks around the MoE layer.

TEST INFRASTRUCTURE ONLY (see the package docstring).

The paper ran a whole MoE decoder at a 4096-token context (Sec. "Experimental Setup": context
length 4096, Flash Attention) but prints no architecture; this follows a Qwen3-MoE-class block.
Per layer l, for the decode token at position p with residual stream x:

1. a = RMSNorm(x) * w_in;  q = W_q a  [Hq x D],  k = W_k a,  v = W_v a  [Hkv x D];
2. per head: q_h = RoPE(RMSNorm(q_h) * w_q, p),  k_g = RoPE(RMSNorm(k_g) * w_k, p);
3. (k_g, v_g) are appended to the layer's KV cache at position p;
4. grouped-query attention over positions 0..p: query head h reads kv head h / (Hq / Hkv),
   o_h = softmax_j(q_h . K_j / sqrt(D)) V;  x = x + W_o [o_0 .. o_{Hq-1}];
5. m = RMSNorm(x) * w_post;  x = x + MoE_l(m), the MoE layer of the package oracle (routing on m,
   one residency step of the shared slot group, experts from the slot copies, combine).

The stack is chained: layer l + 1 routes on what layer l produced, so the residency sees real
cross-layer dependence. All arithmetic is fp64 on the exactly widened stored weights and cache.
"""
from __future__ import annotations

from dataclasses import dataclass

import numpy as np

from . import Oracle, _p, lib, matvec, widen


def rmsnorm(x: np.ndarray, w: np.ndarray, eps: float) -> np.ndarray:
    x = np.ascontiguousarray(x, dtype=np.float64)
    w = np.ascontiguousarray(w, dtype=np.float64)
    out = np.empty_like(x)
    lib().orc_rmsnorm(_p(x), _p(w), x.size, eps, _p(out))
    return out


def rope(x: np.ndarray, pos: int, theta: float) -> np.ndarray:
    x = np.ascontiguousarray(x, dtype=np.float64)
    out = np.empty_like(x)
    lib().orc_rope(_p(x), x.size, pos, theta, _p(out))
    return out


def attend(q: np.ndarray, K: np.ndarray, V: np.ndarray, T: int) -> np.ndarray:
    """q [Hq x D]; K, V [Hkv x Tmax x D] with positions 0..T-1 valid -> out [Hq x D]."""
    q = np.ascontiguousarray(q, dtype=np.float64)
    K = np.ascontiguousarray(K, dtype=np.float64)
    V = np.ascontiguousarray(V, dtype=np.float64)
    Hq, D = q.shape
    Hkv, Tmax, _ = K.shape
    assert Hq % Hkv == 0 and 1 <= T <= Tmax and V.shape == K.shape
    out = np.empty((Hq, D), dtype=np.float64)
    scratch = np.empty(T, dtype=np.float64)
    lib().orc_attend(_p(q), _p(K), _p(V), Hq, Hkv, T, Tmax, D, _p(out), _p(scratch))
    return out


@dataclass
class DecoderStep:
    out: np.ndarray  # f64 [d]: the residual stream after the last layer
    attn: np.ndarray  # f64 [L x d]: W_o o of each layer
    moe_in: np.ndarray  # f64 [L x d]: m, the MoE layer's input
    moe_out: np.ndarray  # f64 [L x d]
    idx: np.ndarray  # int32 [L x k]
    gate: np.ndarray  # f64 [L x k]
    z: np.ndarray  # f64 [L x E]
    records: np.ndarray  # residency records of every layer-step, layer order


class DecoderOracle:
    """Batch-1 decode through dw's chained stack, starting after dw.ctx cached positions.

    layers: None (every layer), or the layers whose attention weights and KV caches are built;
    attention() then serves only those, and decode_token() needs them all. This keeps checks of
    sampled layers of a large stack cheap; the arithmetic is the same."""

    def __init__(self, dw, cap_slots=None, policy="lru", keep_slot_copies=True, max_tokens=None, moe=None,
                 layers=None):
        import synth

        self.dw = dw
        wl = dw.moe
        self.L, self.d = wl.n_layers, wl.d
        self.Hq, self.Hkv, self.D = dw.n_heads, dw.n_kv_heads, dw.head_dim
        self.moe = moe if moe is not None else Oracle.for_workload(
            wl, cap_slots=cap_slots, keep_slot_copies=keep_slot_copies, policy=policy)
        wdt = "fp32" if wl.wdtype == "fp32" else "bf16"
        qd, kd = self.Hq * self.D, self.Hkv * self.D
        self.layers = list(range(self.L)) if layers is None else sorted(set(int(l) for l in layers))
        self.attn_w = {}
        for l in self.layers:
            a = synth.attention_weights(dw, l)
            self.attn_w[l] = {
                "wq": widen(wdt, a["wq"], qd, wl.d), "wk": widen(wdt, a["wk"], kd, wl.d),
                "wv": widen(wdt, a["wv"], kd, wl.d), "wo": widen(wdt, a["wo"], wl.d, qd),
                **{n: _widen_vec(wdt, a[n]) for n in ("norm_in", "norm_post", "norm_q", "norm_k")}}
        self.Tmax = dw.ctx + (wl.tokens if max_tokens is None else max_tokens)
        self.K, self.V = {}, {}
        for l in self.layers:
            K, V = synth.kv_prefix(dw, l)
            self.K[l] = np.zeros((self.Hkv, self.Tmax, self.D), dtype=np.float64)
            self.V[l] = np.zeros_like(self.K[l])
            self.K[l][:, :dw.ctx] = synth.act_to_f64(K, wl.adtype)
            self.V[l][:, :dw.ctx] = synth.act_to_f64(V, wl.adtype)
        self.pos = dw.ctx

    def attention(self, l: int, x: np.ndarray) -> np.ndarray:
        """Steps 1-4 for layer l at the current position: appends to the cache, returns W_o o."""
        w, dw, D = self.attn_w[l], self.dw, self.D
        a = rmsnorm(x, w["norm_in"], dw.eps)
        q = matvec(w["wq"], a).reshape(self.Hq, D)
        k = matvec(w["wk"], a).reshape(self.Hkv, D)
        v = matvec(w["wv"], a).reshape(self.Hkv, D)
        q = np.stack([rope(rmsnorm(q[h], w["norm_q"], dw.eps), self.pos, dw.rope_theta) for h in range(self.Hq)])
        k = np.stack([rope(rmsnorm(k[g], w["norm_k"], dw.eps), self.pos, dw.rope_theta) for g in range(self.Hkv)])
        self.K[l][:, self.pos] = k
        self.V[l][:, self.pos] = v
        o = attend(q, self.K[l], self.V[l], self.pos + 1)
        return matvec(w["wo"], o.reshape(-1))

    def decode_token(self, x0: np.ndarray) -> DecoderStep:
        """One decode token: x0 [d] (fp64 values) enters layer 0."""
        if self.pos >= self.Tmax:
            raise RuntimeError("KV cache full")
        if len(self.layers) != self.L:
            raise RuntimeError("decode_token needs every layer (built with layers=None)")
        L, d, k, E = self.L, self.d, self.moe.k, self.moe.E
        x = np.array(x0, dtype=np.float64)
        attn = np.empty((L, d))
        moe_in = np.empty((L, d))
        moe_out = np.empty((L, d))
        idx = np.empty((L, k), dtype=np.int32)
        gate = np.empty((L, k))
        z = np.empty((L, E))
        recs = []
        for l in range(L):
            attn[l] = self.attention(l, x)
            x = x + attn[l]
            moe_in[l] = rmsnorm(x, self.attn_w[l]["norm_post"], self.dw.eps)
            o, ii, gg, zz, r = self.moe.layer_step(l, moe_in[l][None, :])
            idx[l], gate[l], z[l] = ii[0], gg[0], zz[0]
            recs.append(r)
            moe_out[l] = o[0]
            x = x + moe_out[l]
        self.moe.token_step += 1
        self.pos += 1
        return DecoderStep(x, attn, moe_in, moe_out, idx, gate, z, np.concatenate(recs))


def _widen_vec(dt: str, raw: np.ndarray) -> np.ndarray:
    return widen(dt, raw.reshape(1, -1), 1, raw.size).reshape(-1)
