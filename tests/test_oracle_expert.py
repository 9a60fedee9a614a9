"""Pins of the oracle's expert FFN, combine and weight widening (MoE sub-modules, paper
Section "Related Work" / "Rotary GPU Concept": experts are the units of residency).

Checked against: numpy float64 matmuls (an independent library routine), pure-Python
loops, closed forms (W_g = 0 -> 0; one-hot inputs pick columns), known bf16 bit
patterns, hand-packed int4 bytes, and exact int4 round trips.
"""
import math

import numpy as np
import pytest

import oracle
import synth
from oracle.brute import expert_brute


def _np_expert(Wg, Wu, Wd, x):
    a = Wg @ x
    return Wd @ (a / (1 + np.exp(-a)) * (Wu @ x))


@pytest.mark.parametrize("seed", range(4))
def test_expert_matches_numpy_on_tiny_config_shapes(seed):
    wl = synth.WORKLOADS["tiny_fp32"]
    w = synth.expert_weights(wl, 0, seed)
    Wg, Wu, Wd = (np.asarray(a, dtype=np.float64) for a in (w.gate, w.up, w.down))
    x = synth.act_to_f64(synth.hidden_stream(wl, 0, 0, 3)[seed % 3], "fp32")
    y, u = oracle.expert_ffn(Wg, Wu, Wd, x)
    np.testing.assert_allclose(y, _np_expert(Wg, Wu, Wd, x), rtol=1e-11, atol=1e-13)
    a = Wg @ x
    np.testing.assert_allclose(u, a / (1 + np.exp(-a)) * (Wu @ x), rtol=1e-11, atol=1e-14)


def test_expert_matches_python_loops():
    rng = np.random.default_rng(2)
    d, I = 12, 7
    Wg, Wu, Wd = rng.standard_normal((I, d)), rng.standard_normal((I, d)), rng.standard_normal((d, I))
    x = rng.standard_normal(d)
    y, _ = oracle.expert_ffn(Wg, Wu, Wd, x)
    np.testing.assert_allclose(y, expert_brute(Wg.tolist(), Wu.tolist(), Wd.tolist(), x.tolist()), rtol=1e-13)


def test_zero_gate_weights_give_zero_output():
    rng = np.random.default_rng(3)
    d, I = 16, 8
    y, u = oracle.expert_ffn(np.zeros((I, d)), rng.standard_normal((I, d)), rng.standard_normal((d, I)),
                             rng.standard_normal(d))
    assert np.all(u == 0) and np.all(y == 0)


def test_one_hot_input_combines_columns():
    rng = np.random.default_rng(4)
    d, I, j = 10, 6, 3
    Wg, Wu, Wd = rng.standard_normal((I, d)), rng.standard_normal((I, d)), rng.standard_normal((d, I))
    x = np.zeros(d)
    x[j] = 1.0
    y, _ = oracle.expert_ffn(Wg, Wu, Wd, x)
    coef = [Wg[i, j] / (1 + math.exp(-Wg[i, j])) * Wu[i, j] for i in range(I)]
    expect = sum(coef[i] * Wd[:, i] for i in range(I))
    np.testing.assert_allclose(y, expect, rtol=1e-13)


def test_silu_limits():
    # a = 0 -> u = 0; large a -> silu(a) ~ a; very negative a -> ~0
    Wg = np.array([[0.0], [40.0], [-800.0]])
    Wu = np.ones((3, 1))
    Wd = np.eye(3)
    y, u = oracle.expert_ffn(Wg, Wu, Wd, np.array([1.0]))
    assert u[0] == 0.0
    assert abs(u[1] - 40.0) < 1e-12
    assert u[2] == 0.0 or abs(u[2]) < 1e-300


def test_combine_is_gate_weighted_sum_in_rank_order():
    rng = np.random.default_rng(5)
    y = rng.standard_normal((8, 32))
    g = rng.random(8)
    np.testing.assert_allclose(oracle.combine(y, g), g @ y, rtol=1e-13)
    # sequential rank order: identical to an explicit left fold
    fold = np.zeros(32)
    for r in range(8):
        fold = fold + g[r] * y[r]
    np.testing.assert_array_equal(oracle.combine(y, g), fold)


def test_widen_bf16_known_patterns():
    bits = np.array([[0x3F80, 0xBF80, 0x4049, 0x0000, 0x8000, 0x7F80, 0x3E00, 0x0001]], dtype=np.uint16)
    w = oracle.widen("bf16", bits, 1, 8)
    assert w[0, :5].tolist() == [1.0, -1.0, 3.140625, 0.0, 0.0]
    assert math.copysign(1.0, w[0, 4]) == -1.0
    assert math.isinf(w[0, 5]) and w[0, 6] == 0.125
    assert w[0, 7] == 2.0 ** -133


def test_widen_int4_hand_packed():
    # row of 128: byte 0 = 0x9F -> elements 0 (low nibble 0xF = -1) and 1 (high 0x9 = -7);
    # byte 1 = 0x70 -> elements 2 (0) and 3 (7); scale bf16 0x3F00 = 0.5
    q = np.zeros((1, 64), dtype=np.uint8)
    q[0, 0], q[0, 1], q[0, 63] = 0x9F, 0x70, 0x18
    s = np.array([[0x3F00]], dtype=np.uint16)
    w = oracle.widen("int4", q, 1, 128, s)
    assert w[0, :4].tolist() == [-0.5, -3.5, 0.0, 3.5]
    assert w[0, 126] == -4.0 and w[0, 127] == 0.5
    assert np.count_nonzero(w) == 5


def test_int4_round_trip_is_exact_for_representable_weights():
    rng = np.random.default_rng(6)
    rows, cols = 5, 256
    q = rng.integers(-7, 8, size=(rows, cols))
    q[:, ::128] = 7  # each group reaches absmax = 7 s exactly
    s = synth.bf16_bits_to_f32(synth.f32_to_bf16_bits(rng.uniform(0.01, 0.2, size=(rows, 2))))
    w = (q * np.repeat(s, 128, axis=1)).astype(np.float32)
    qp, sb = synth.quant_int4_g128(w)
    np.testing.assert_array_equal(oracle.widen("int4", qp, rows, cols, sb), w.astype(np.float64))


def test_int4_dequant_error_bound_on_normal_weights():
    wl = synth.WORKLOADS["stack48_int4"]
    rng = np.random.default_rng(8)
    w = (rng.standard_normal((64, 2048)) / math.sqrt(2048)).astype(np.float32)
    qp, sb = synth.quant_int4_g128(w)
    deq = oracle.widen("int4", qp, 64, 2048, sb)
    s = np.repeat(synth.bf16_bits_to_f32(sb).astype(np.float64), 128, axis=1)
    amax = np.repeat(np.abs(w.reshape(64, 16, 128)).max(axis=2), 128, axis=1).astype(np.float64)
    bound = 0.5 * s + np.maximum(amax - 7 * s, 0) + 1e-12
    assert np.all(np.abs(deq - w) <= bound)
    assert wl.wdtype == "int4"
