"""Pins of the oracle's routing result (paper Fig. 1: the routing result h, r drives residency).

Checked against: a pure-Python brute force that sorts the full softmax explicitly,
the closed form "renormalised top-k gates = softmax of the top-k logits", the
invariant sum(g) = 1, the special case k = E (gates = full softmax), crafted ties,
and softmax's shift invariance / overflow behaviour.
"""
import math

import numpy as np
import pytest

import oracle
from oracle.brute import router_brute


def _rand(seed, E, d):
    rng = np.random.default_rng(seed)
    return rng.standard_normal((E, d)) / math.sqrt(d), rng.standard_normal(d)


@pytest.mark.parametrize("seed", range(6))
@pytest.mark.parametrize("E,d,k", [(8, 16, 1), (8, 16, 2), (8, 16, 3), (8, 16, 8), (13, 7, 5), (32, 24, 8)])
def test_router_matches_brute_force(seed, E, d, k):
    Wr, h = _rand(seed, E, d)
    idx, gate, z, p = oracle.router(Wr, h, k)
    sel, g, zb, pb = router_brute(Wr.tolist(), h.tolist(), k)
    assert list(idx) == sel
    np.testing.assert_allclose(gate, g, rtol=1e-12, atol=0)
    np.testing.assert_allclose(z, zb, rtol=1e-12, atol=1e-15)
    np.testing.assert_allclose(p, pb, rtol=1e-12, atol=0)


@pytest.mark.parametrize("seed", range(10))
def test_gates_sum_to_one(seed):
    Wr, h = _rand(seed, 128, 64)
    _, gate, _, _ = oracle.router(Wr, h, 8)
    assert abs(gate.sum() - 1.0) <= 1e-12
    assert np.all(gate > 0)
    assert np.all(np.diff(gate) <= 0), "gates follow descending logits"


@pytest.mark.parametrize("seed", range(10))
def test_renorm_gates_equal_softmax_over_selected_logits(seed):
    Wr, h = _rand(seed, 64, 32)
    idx, gate, z, _ = oracle.router(Wr, h, 6)
    zs = z[idx]
    closed = np.exp(zs - zs.max()) / np.exp(zs - zs.max()).sum()
    np.testing.assert_allclose(gate, closed, rtol=1e-13)


def test_k_equals_E_gives_full_softmax_in_sorted_order():
    Wr, h = _rand(3, 16, 8)
    idx, gate, z, p = oracle.router(Wr, h, 16)
    assert sorted(idx.tolist()) == list(range(16))
    np.testing.assert_allclose(gate, p[idx], rtol=1e-13)
    assert np.all(np.diff(z[idx]) <= 0)


def test_topk_selects_largest_logits_descending():
    Wr, h = _rand(5, 128, 2048)
    idx, _, z, _ = oracle.router(Wr, h, 8)
    order = np.lexsort((np.arange(128), -z))
    assert idx.tolist() == order[:8].tolist()


def test_ties_break_toward_lower_id():
    # rows 2, 5 and 6 identical -> equal logits; row 3 strictly larger
    d = 4
    Wr = np.zeros((8, d))
    Wr[:, 0] = [-1, -2, 0.5, 2.0, -3, 0.5, 0.5, -0.25]
    h = np.array([1.0, 0.0, 0.0, 0.0])
    idx, gate, _, _ = oracle.router(Wr, h, 3)
    assert idx.tolist() == [3, 2, 5]
    idx4, _, _, _ = oracle.router(Wr, h, 4)
    assert idx4.tolist() == [3, 2, 5, 6]
    assert gate[1] == gate[2]


def test_no_renorm_returns_raw_probabilities():
    Wr, h = _rand(9, 32, 16)
    idx, gate, _, p = oracle.router(Wr, h, 4, renorm=False)
    np.testing.assert_array_equal(gate, p[idx])
    assert gate.sum() < 1.0


def test_forced_ids_reweight_over_forced_set():
    Wr, h = _rand(11, 32, 16)
    forced = np.array([7, 1, 30], dtype=np.int32)
    idx, gate, _, p = oracle.router(Wr, h, 3, forced_idx=forced)
    assert idx.tolist() == [7, 1, 30]
    np.testing.assert_allclose(gate, p[forced] / p[forced].sum(), rtol=1e-13)


def test_softmax_shift_invariance_and_no_overflow():
    z = np.array([1000.0, 1000.0, 999.0])
    p = oracle.softmax(z)
    e = math.exp(-1.0)
    np.testing.assert_allclose(p, [1 / (2 + e), 1 / (2 + e), e / (2 + e)], rtol=1e-14)
    z2 = np.array([0.3, -1.2, 2.5, 0.0])
    np.testing.assert_allclose(oracle.softmax(z2), oracle.softmax(z2 + 123.0), rtol=1e-12)


def test_matvec_matches_numpy():
    rng = np.random.default_rng(0)
    W = rng.standard_normal((37, 53))
    x = rng.standard_normal(53)
    np.testing.assert_allclose(oracle.matvec(W, x), W @ x, rtol=1e-12, atol=1e-13)
