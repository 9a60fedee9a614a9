"""Pins of the oracle's decoder block around the MoE layer (RMSNorm, rotary positions, grouped-query
attention over a KV cache, the chained residual stream).

Checked against: pure-Python restatements (a loop RMSNorm, rotary embedding as complex
multiplication, attention with explicit loops), closed forms and invariants (norm preservation,
relative positions, one-hot rotation, single-position and uniform attention, grouped-query
attention equal to multi-head attention with repeated kv heads), and for the whole block: a
matrix-form evaluation of the stack over a token sequence with a causal mask (no KV cache, no
residency), the cap invariance, and the residency trace against an independent recency list.
"""
import numpy as np
import pytest

import oracle
import synth
from oracle.brute import RecencyListLRU, attend_brute, rmsnorm_brute, rope_brute
from oracle.decoder import DecoderOracle, attend, rmsnorm, rope


# ---- RMSNorm

@pytest.mark.parametrize("seed", range(4))
def test_rmsnorm_matches_loop(seed):
    rng = np.random.default_rng(seed)
    x, w = rng.standard_normal(37), rng.standard_normal(37)
    np.testing.assert_allclose(rmsnorm(x, w, 1e-6), rmsnorm_brute(list(x), list(w), 1e-6), rtol=1e-13, atol=0)


def test_rmsnorm_closed_form_and_scale_invariance():
    n, c, eps = 64, -3.0, 1e-2
    np.testing.assert_allclose(rmsnorm(np.full(n, c), np.ones(n), eps), np.full(n, c / np.sqrt(c * c + eps)),
                               rtol=1e-15)
    x = np.random.default_rng(1).standard_normal(100)
    y = rmsnorm(x, np.ones(100), 0.0)
    np.testing.assert_allclose(np.sqrt(np.mean(y * y)), 1.0, rtol=1e-14)
    np.testing.assert_allclose(rmsnorm(7.5 * x, np.ones(100), 0.0), y, rtol=1e-14)


# ---- rotary positions

@pytest.mark.parametrize("pos", [0, 1, 17, 4095, 100_000])
def test_rope_matches_complex_rotation(pos):
    x = np.random.default_rng(pos % 7).standard_normal(64)
    np.testing.assert_allclose(rope(x, pos, 1e6), rope_brute(list(x), pos, 1e6), rtol=1e-12, atol=1e-12)


def test_rope_identity_norm_and_one_hot():
    D, theta = 128, 1e6
    x = np.random.default_rng(3).standard_normal(D)
    np.testing.assert_array_equal(rope(x, 0, theta), x)
    np.testing.assert_allclose(np.linalg.norm(rope(x, 1234, theta)), np.linalg.norm(x), rtol=1e-14)
    for i in (0, 5, D // 2 - 1):
        e = np.zeros(D)
        e[i] = 1.0
        a = 77 * theta ** (-2.0 * i / D)
        want = np.zeros(D)
        want[i], want[i + D // 2] = np.cos(a), np.sin(a)
        np.testing.assert_allclose(rope(e, 77, theta), want, atol=1e-15)


def test_rope_scores_depend_on_relative_position_only():
    rng = np.random.default_rng(4)
    q, k = rng.standard_normal(128), rng.standard_normal(128)
    for p, s, shift in ((10, 3, 500), (4000, 0, 95), (1, 2, 7)):
        a = rope(q, p, 1e6) @ rope(k, s, 1e6)
        b = rope(q, p + shift, 1e6) @ rope(k, s + shift, 1e6)
        np.testing.assert_allclose(a, b, rtol=1e-10)
    np.testing.assert_allclose(rope(rope(q, 40, 1e6), 60, 1e6), rope(q, 100, 1e6), rtol=1e-12, atol=1e-12)


# ---- attention

@pytest.mark.parametrize("Hq,Hkv,T", [(4, 2, 5), (4, 4, 1), (6, 2, 9), (2, 1, 3)])
def test_attention_matches_loops(Hq, Hkv, T):
    rng = np.random.default_rng(Hq * 10 + T)
    D, Tmax = 16, T + 3
    q = rng.standard_normal((Hq, D))
    K, V = rng.standard_normal((Hkv, Tmax, D)), rng.standard_normal((Hkv, Tmax, D))
    want = attend_brute(q.tolist(), K.tolist(), V.tolist(), T)
    np.testing.assert_allclose(attend(q, K, V, T), want, rtol=1e-12, atol=1e-14)


def test_attention_special_cases():
    rng = np.random.default_rng(9)
    Hq, Hkv, D, Tmax = 4, 2, 8, 6
    K, V = rng.standard_normal((Hkv, Tmax, D)), rng.standard_normal((Hkv, Tmax, D))
    q = rng.standard_normal((Hq, D))
    # one position: every head returns its kv head's value row
    out = attend(q, K, V, 1)
    for h in range(Hq):
        np.testing.assert_allclose(out[h], V[h // 2, 0], rtol=1e-15)
    # zero query: uniform weights, the mean of the value rows
    out = attend(np.zeros((Hq, D)), K, V, 5)
    for h in range(Hq):
        np.testing.assert_allclose(out[h], V[h // 2, :5].mean(axis=0), rtol=1e-13)
    # a dominant score: the arg-max position's value row, finite despite huge logits
    qq = np.zeros((Hq, D))
    qq[:, 0] = 1e4
    Kd = K.copy()
    Kd[:, 3, 0] = 10.0
    Kd[:, [0, 1, 2, 4], 0] = 0.0
    out = attend(qq, Kd, V, 5)
    assert np.isfinite(out).all()
    np.testing.assert_allclose(out[0], V[0, 3], rtol=1e-12)


def test_grouped_query_equals_multi_head_with_repeated_kv():
    rng = np.random.default_rng(11)
    Hq, Hkv, D, T = 8, 2, 16, 7
    q = rng.standard_normal((Hq, D))
    K, V = rng.standard_normal((Hkv, T, D)), rng.standard_normal((Hkv, T, D))
    Krep, Vrep = np.repeat(K, Hq // Hkv, axis=0), np.repeat(V, Hq // Hkv, axis=0)
    np.testing.assert_allclose(attend(q, K, V, T), attend(q, Krep, Vrep, T), rtol=1e-15)


def test_attention_is_invariant_to_the_order_of_cached_positions():
    rng = np.random.default_rng(12)
    q = rng.standard_normal((4, 16))
    K, V = rng.standard_normal((2, 9, 16)), rng.standard_normal((2, 9, 16))
    perm = rng.permutation(9)
    np.testing.assert_allclose(attend(q, K, V, 9), attend(q, K[:, perm], V[:, perm], 9), rtol=1e-13)


# ---- the chained block

DW = synth.DECODERS["tiny_block_fp32"]


def _inputs(dw, T):
    return synth.act_to_f64(synth.token_inputs(dw, T), dw.moe.adtype)


def _matrix_form(dw, X):
    """The whole stack over a token sequence at once: rows of X are consecutive positions after the
    cached prefix; causal attention over prefix + sequence with a mask; experts read straight from
    the host tier (no residency). Independent of the incremental KV-cache evaluation."""
    wl = dw.moe
    T, d = X.shape
    Hq, Hkv, D, c = dw.n_heads, dw.n_kv_heads, dw.head_dim, dw.ctx
    X = X.copy()
    for l in range(wl.n_layers):
        a = synth.attention_weights(dw, l)
        W = {n: a[n].astype(np.float64) for n in a}  # fp32 storage: exact
        nrm = lambda M, w: M / np.sqrt((M * M).mean(axis=-1, keepdims=True) + dw.eps) * w  # noqa: E731
        A = nrm(X, W["norm_in"])
        Q = (A @ W["wq"].T).reshape(T, Hq, D)
        Kn = (A @ W["wk"].T).reshape(T, Hkv, D)
        Vn = (A @ W["wv"].T).reshape(T, Hkv, D)
        Q, Kn = nrm(Q, W["norm_q"]), nrm(Kn, W["norm_k"])
        pos = c + np.arange(T)
        ang = pos[:, None] * dw.rope_theta ** (-2.0 * np.arange(D // 2) / D)[None, :]  # [T x D/2]
        rot = lambda M: np.concatenate([M[..., :D // 2] * np.cos(ang)[:, None] - M[..., D // 2:] * np.sin(ang)[:, None],  # noqa: E731
                                        M[..., D // 2:] * np.cos(ang)[:, None] + M[..., :D // 2] * np.sin(ang)[:, None]],
                                       axis=-1)
        Q, Kn = rot(Q), rot(Kn)
        Kp, Vp = (v.astype(np.float64) for v in synth.kv_prefix(dw, l))  # [Hkv x c x D]
        Kall = np.concatenate([Kp, Kn.transpose(1, 0, 2)], axis=1)  # [Hkv x (c+T) x D]
        Vall = np.concatenate([Vp, Vn.transpose(1, 0, 2)], axis=1)
        O = np.empty((T, Hq, D))
        for h in range(Hq):
            g = h // (Hq // Hkv)
            S = Q[:, h, :] @ Kall[g].T / np.sqrt(D)  # [T x (c+T)]
            S[np.arange(c + T)[None, :] > (c + np.arange(T))[:, None]] = -np.inf
            P = np.exp(S - S.max(axis=1, keepdims=True))
            P /= P.sum(axis=1, keepdims=True)
            O[:, h, :] = P @ Vall[g]
        X = X + O.reshape(T, Hq * D) @ W["wo"].T
        M = nrm(X, W["norm_post"])
        Wr = synth.router_weights(wl, l).astype(np.float64)
        for t in range(T):
            z = Wr @ M[t]
            sel = sorted(range(wl.n_experts), key=lambda e: (-z[e], e))[:wl.top_k]
            p = np.exp(z[sel] - z[sel].max())
            p /= p.sum()
            y = np.zeros(d)
            for r, e in enumerate(sel):
                ew = synth.expert_weights(wl, l, e)
                Wg, Wu, Wd = (m.astype(np.float64) for m in (ew.gate, ew.up, ew.down))
                g_, u_ = Wg @ M[t], Wu @ M[t]
                y += p[r] * (Wd @ (g_ / (1.0 + np.exp(-g_)) * u_))
            X[t] = X[t] + y
    return X


def test_incremental_decode_equals_the_matrix_form():
    T = 6
    X0 = _inputs(DW, T)
    dec = DecoderOracle(DW, max_tokens=T)
    got = np.stack([dec.decode_token(X0[t]).out for t in range(T)])
    np.testing.assert_allclose(got, _matrix_form(DW, X0), rtol=1e-10, atol=1e-10)


def test_zero_output_projections_pass_the_stream_through():
    wl = DW.moe

    def zero_down(l, e):
        w = synth.expert_weights(wl, l, e)
        w.down = np.zeros_like(w.down)
        return w

    moe = oracle.Oracle.for_workload(wl, experts=zero_down)
    dec = DecoderOracle(DW, moe=moe, max_tokens=3)
    for a in dec.attn_w.values():
        a["wo"][:] = 0.0
    X0 = _inputs(DW, 3)
    for t in range(3):
        np.testing.assert_array_equal(dec.decode_token(X0[t]).out, X0[t])


def test_outputs_do_not_depend_on_the_cap_and_the_trace_is_lru():
    T = 8
    X0 = _inputs(DW, T)
    n_gid = DW.moe.n_gid
    capped, full = DecoderOracle(DW, max_tokens=T), DecoderOracle(DW, cap_slots=n_gid, max_tokens=T)
    ref = RecencyListLRU(DW.moe.cap_slots)
    E = DW.moe.n_experts
    for t in range(T):
        a, b = capped.decode_token(X0[t]), full.decode_token(X0[t])
        np.testing.assert_array_equal(a.out, b.out)
        np.testing.assert_array_equal(a.idx, b.idx)
        expect = []
        for l in range(DW.moe.n_layers):
            expect += ref.step([l * E + int(e) for e in a.idx[l]])
        got = [(int(r["layer"]) * E + int(r["expert"]), int(r["kind"]), int(r["slot"]), int(r["evicted"]))
               for r in a.records]
        assert got == expect
    assert int((capped.moe.table.gid_of >= 0).sum()) == DW.moe.cap_slots


def test_the_cache_grows_by_one_position_per_token_and_refuses_overflow():
    dec = DecoderOracle(DW, max_tokens=2)
    X0 = _inputs(DW, 3)
    assert dec.pos == DW.ctx
    dec.decode_token(X0[0])
    dec.decode_token(X0[1])
    assert dec.pos == DW.ctx + 2
    assert all(np.abs(dec.K[l][:, DW.ctx:DW.ctx + 2]).sum() > 0 for l in dec.layers)
    with pytest.raises(RuntimeError):
        dec.decode_token(X0[2])


def test_a_subset_of_layers_gives_the_same_attention_as_the_whole_stack():
    # built for layers 0 and 1 only, the oracle's attention of those layers on the same inputs is
    # bit-identical to the full oracle's; decode_token refuses to run on a subset
    X0 = _inputs(DW, 2)
    full = DecoderOracle(DW)
    part = DecoderOracle(DW, layers=[1, 0])
    assert part.layers == [0, 1]
    for t in range(2):
        r = full.decode_token(X0[t])
        x = np.array(X0[t], dtype=np.float64)
        for l in range(DW.moe.n_layers):
            np.testing.assert_array_equal(part.attention(l, x), r.attn[l])
            x = x + r.attn[l] + r.moe_out[l]
        part.pos += 1
    one = DecoderOracle(DW, layers=[0])
    with pytest.raises(RuntimeError):
        one.decode_token(X0[0])
