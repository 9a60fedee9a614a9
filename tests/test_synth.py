"""The seeded input generator shared by the oracle and the CUDA path (it holds none of the
method's arithmetic): counter-based normals independent of how they are sliced, bf16 rounding to
nearest even, the int4 g128 quantisation rules, the AR(1) recurrence, and the layouts the decode
step takes."""
import math

import numpy as np
import pytest

import synth


def test_normals_do_not_depend_on_slicing():
    full = synth.normal(7, 3, 0, 1001)
    for start, n in [(0, 1), (1, 1), (1, 10), (5, 7), (500, 501), (999, 2)]:
        np.testing.assert_array_equal(synth.normal(7, 3, start, n), full[start:start + n])


def test_normals_are_reproducible_and_streams_differ():
    a = synth.normal(1, 2, 0, 4096)
    np.testing.assert_array_equal(a, synth.normal(1, 2, 0, 4096))
    assert not np.array_equal(a, synth.normal(1, 3, 0, 4096))
    assert not np.array_equal(a, synth.normal(2, 2, 0, 4096))


def test_normal_moments():
    x = synth.normal(0, 11, 0, 1 << 20).astype(np.float64)
    assert abs(x.mean()) < 5e-3
    assert abs(x.std() - 1.0) < 5e-3
    assert abs(np.mean(x ** 3)) < 1e-2 and abs(np.mean(x ** 4) - 3.0) < 3e-2
    y = synth.normal(0, 11, 0, 1000, std=0.25)
    np.testing.assert_allclose(y, 0.25 * x[:1000].astype(np.float32), rtol=1e-6)


def _bf16_rne(x):
    """Plain reimplementation: keep the top 16 bits after adding 0x7fff plus the lowest kept bit."""
    u = np.asarray(x, dtype=np.float32).view(np.uint32).astype(np.uint64)
    r = (u + 0x7FFF + ((u >> 16) & 1)) >> 16
    return r.astype(np.uint16)


def test_bf16_rounding_is_nearest_even():
    rng = np.random.default_rng(0)
    x = (rng.standard_normal(100000) * 10.0 ** rng.integers(-20, 20, 100000)).astype(np.float32)
    np.testing.assert_array_equal(synth.f32_to_bf16_bits(x), _bf16_rne(x))
    # exact halfway cases go to the even neighbour
    one = np.float32(1.0).view(np.uint32)
    up = np.array([one | 0x8000, (one + 0x10000) | 0x8000], dtype=np.uint32).view(np.float32)
    assert synth.f32_to_bf16_bits(up).tolist() == [0x3F80, 0x3F82]
    # NaN stays NaN, infinities stay infinite
    nan = synth.bf16_bits_to_f32(synth.f32_to_bf16_bits(np.array([np.nan], dtype=np.float32)))
    assert np.isnan(nan[0])
    inf = synth.bf16_bits_to_f32(synth.f32_to_bf16_bits(np.array([np.inf, -np.inf], dtype=np.float32)))
    assert inf.tolist() == [np.inf, -np.inf]


def test_int4_quantisation_rules():
    rng = np.random.default_rng(1)
    w = rng.standard_normal((3, 256)).astype(np.float32)
    w[1, 128:] = 0.0  # an all-zero group: scale 0, every q 0
    q, s = synth.quant_int4_g128(w)
    for r in range(3):
        for g in range(2):
            grp = w[r, 128 * g:128 * (g + 1)]
            scale_bits = synth.f32_to_bf16_bits(np.array([np.abs(grp).max() / np.float32(7.0)], dtype=np.float32))[0]
            assert s[r, g] == scale_bits
            scale = synth.bf16_bits_to_f32(np.array([scale_bits]))[0]
            for i in range(128):
                c = 128 * g + i
                byte = int(q[r, c // 2])
                nib = byte & 0xF if c % 2 == 0 else byte >> 4
                qv = nib - 16 if nib >= 8 else nib
                want = 0 if scale == 0 else int(np.clip(np.rint(grp[i] / scale), -7, 7))
                assert qv == want, (r, c)
    with pytest.raises(ValueError):
        synth.quant_int4_g128(np.zeros((2, 100), dtype=np.float32))


def test_ar1_recurrence_and_stationary_variance():
    T, d, rho = 50, 64, 0.8
    h = synth.ar1(5, 9, T, d, rho)
    eps = synth.normal(5, 9, 0, T * d).astype(np.float64).reshape(T, d)
    np.testing.assert_array_equal(h[0], eps[0])
    c = math.sqrt(1.0 - rho * rho)
    for t in range(1, T):
        np.testing.assert_array_equal(h[t], rho * h[t - 1] + c * eps[t])
    long = synth.ar1(5, 10, 4000, 64, rho)
    assert abs(long[100:].var() - 1.0) < 0.1


def test_hidden_layout_and_rounding():
    wl = synth.WORKLOADS["tiny_fp32"].replace(n_layers=2, batch=3, tokens=5)
    h = synth.hidden_all(wl)
    assert h.shape == (5, 2, 3, wl.d) and h.dtype == np.float32
    for l in range(2):
        for b in range(3):
            np.testing.assert_array_equal(h[:, l, b], synth.hidden_stream(wl, l, b))
    assert not np.array_equal(h[:, 0, 0], h[:, 0, 1])  # each sequence has its own stream
    wb = wl.replace(wdtype="bf16", adtype="bf16")
    hb = synth.hidden_all(wb)
    assert hb.dtype == np.uint16
    # bf16 inputs are the fp32 values rounded once more (fp64 -> fp32 -> bf16)
    np.testing.assert_array_equal(hb, synth.f32_to_bf16_bits(h))


def test_weight_shapes_and_scale():
    wl = synth.WORKLOADS["stack48_int4"]
    w = synth.expert_weights(wl, 3, 17)
    assert w.gate.shape == (wl.d_ff, wl.d // 2) and w.down.shape == (wl.d, wl.d_ff // 2)
    assert w.s_gate.shape == (wl.d_ff, wl.d // 128) and w.s_down.shape == (wl.d, wl.d_ff // 128)
    wb = synth.WORKLOADS["layer_bf16"]
    r = synth.bf16_bits_to_f32(synth.router_weights(wb, 0)).astype(np.float64)
    assert r.shape == (wb.n_experts, wb.d)
    assert abs(r.std() * math.sqrt(wb.d) - 1.0) < 0.01  # std = 1 / sqrt(fan_in)


def test_decoder_inputs_shapes_scales_and_independence():
    dw = synth.DECODERS["tiny_block_fp32"]
    wl = dw.moe
    a0, a1 = synth.attention_weights(dw, 0), synth.attention_weights(dw, 1)
    qd, kd = dw.n_heads * dw.head_dim, dw.n_kv_heads * dw.head_dim
    assert a0["wq"].shape == (qd, wl.d) and a0["wk"].shape == (kd, wl.d) and a0["wo"].shape == (wl.d, qd)
    # N(0, 1/fan_in) projections, 1 + N(0, 0.1^2) norm weights
    np.testing.assert_allclose(a0["wq"].std() * np.sqrt(wl.d), 1.0, rtol=0.05)
    np.testing.assert_allclose(a0["wo"].std() * np.sqrt(qd), 1.0, rtol=0.05)
    np.testing.assert_allclose(a0["norm_in"].mean(), 1.0, atol=0.03)
    np.testing.assert_allclose(a0["norm_in"].std(), dw.norm_std, rtol=0.2)
    # layers and matrices draw from different streams; none collides with the router or experts
    assert not np.array_equal(a0["wq"], a1["wq"])
    assert not np.array_equal(a0["wk"][:, :], a0["wv"][:, :])
    r0 = synth.router_weights(wl, 0)
    assert not np.array_equal(a0["wq"][:wl.n_experts], r0)
    K, V = synth.kv_prefix(dw, 0)
    assert K.shape == V.shape == (dw.n_kv_heads, dw.ctx, dw.head_dim)
    assert not np.array_equal(K, V)
    x = synth.token_inputs(dw, 200).astype(np.float64)
    # AR(1): lag-1 correlation rho, unit variance
    c = (x[1:] * x[:-1]).mean() / (x * x).mean()
    np.testing.assert_allclose(c, wl.rho, atol=0.05)
    np.testing.assert_allclose(x.var(), 1.0, atol=0.15)
    np.testing.assert_array_equal(synth.token_inputs(dw, 5), synth.token_inputs(dw, 200)[:5])


def test_decoder_inputs_bf16_storage():
    dw = synth.DECODERS["tiny_block_fp32"].replace(
        moe=synth.WORKLOADS["tiny_fp32"].replace(wdtype="bf16", adtype="bf16", n_layers=2))
    a = synth.attention_weights(dw, 0)
    assert a["wq"].dtype == np.uint16 and a["norm_q"].dtype == np.uint16
    f = synth.attention_weights(synth.DECODERS["tiny_block_fp32"], 0)
    np.testing.assert_array_equal(a["wq"], synth.f32_to_bf16_bits(f["wq"]))
    K, _ = synth.kv_prefix(dw, 1)
    assert K.dtype == np.uint16
