"""Pins of the expert FFN / combine oracle (Section 3.1 Eq. topk and the shared experts).

Naive loops on tiny shapes, the library sigmoid, closed forms (zero weights give zero outputs,
E = K = 1 with renormalised gates is a dense SwiGLU MLP), and linearity in the gates.
"""
import numpy as np
import pytest
import scipy.special

from oracle import ffn as F


def test_silu_values():
    u = np.linspace(-30, 30, 601)
    np.testing.assert_allclose(F.silu(u), u * scipy.special.expit(u), rtol=1e-14, atol=1e-300)
    assert F.silu(0.0) == 0.0
    assert F.silu(-800.0) == 0.0  # exp overflow -> exactly -0
    assert F.silu(50.0) == pytest.approx(50.0, rel=1e-20)


def _naive_expert(x, w1, w3, w2):
    d, w = x.shape[0], w1.shape[0]
    h = []
    for r in range(w):
        g = sum(w1[r, j] * x[j] for j in range(d))
        u = sum(w3[r, j] * x[j] for j in range(d))
        h.append(g / (1.0 + np.exp(-g)) * u)
    return np.array([sum(w2[i, r] * h[r] for r in range(w)) for i in range(d)])


def _experts(g, E, d, w):
    return [(g.standard_normal((w, d)), g.standard_normal((w, d)), g.standard_normal((d, w)))
            for _ in range(E)]


def test_expert_naive_loops_nonsquare():
    g = np.random.default_rng(0)
    d, w = 5, 3  # d != w catches a transposed W2
    x = g.standard_normal((4, d))
    w1, w3, w2 = _experts(g, 1, d, w)[0]
    out = F.expert(x, w1, w3, w2)
    for t in range(4):
        np.testing.assert_allclose(out[t], _naive_expert(x[t], w1, w3, w2), rtol=1e-12)
    # swapping the gate and up projections changes the result (silu is not symmetric)
    assert not np.allclose(F.expert(x, w3, w1, w2), out)


def test_single_expert_is_dense_swiglu():
    g = np.random.default_rng(1)
    d, w = 6, 4
    x = g.standard_normal((7, d))
    ex = _experts(g, 1, d, w)
    y = F.moe_layer(x, np.zeros((7, 1), np.int32), np.ones((7, 1)), ex)
    for t in range(7):
        np.testing.assert_allclose(y[t], _naive_expert(x[t], *ex[0]), rtol=1e-12)


def test_combine_naive():
    g = np.random.default_rng(2)
    E, K, d, w, T = 4, 2, 5, 3, 6
    x = g.standard_normal((T, d))
    ex = _experts(g, E, d, w)
    sh = _experts(g, 2, d, w)
    idx = np.array([[0, 1], [2, 0], [3, 2], [1, 3], [0, 3], [2, 1]], np.int32)
    gate = g.uniform(0, 1, (T, K))
    y = F.moe_layer(x, idx, gate, ex, shared=sh)
    for t in range(T):
        ref = sum(gate[t, k] * _naive_expert(x[t], *ex[idx[t, k]]) for k in range(K))
        ref = ref + sum(_naive_expert(x[t], *s) for s in sh)
        np.testing.assert_allclose(y[t], ref, rtol=1e-11)


def test_zero_cases():
    g = np.random.default_rng(3)
    E, d, w, T = 3, 8, 4, 5
    x = g.standard_normal((T, d))
    ex = [(w1, np.zeros_like(w3), w2) for w1, w3, w2 in _experts(g, E, d, w)]  # W3 = 0 -> h = 0
    idx = np.array([[0, 1]] * T, np.int32)
    assert np.all(F.moe_layer(x, idx, np.ones((T, 2)), ex) == 0)
    ex = _experts(g, E, d, w)
    assert np.all(F.moe_layer(np.zeros((T, d)), idx, np.ones((T, 2)), ex) == 0)
    assert np.all(F.moe_layer(x, idx, np.zeros((T, 2)), ex) == 0)


def test_linear_in_gates():
    g = np.random.default_rng(4)
    E, d, w, T = 3, 8, 4, 5
    x = g.standard_normal((T, d))
    ex = _experts(g, E, d, w)
    idx = np.array([[0, 2]] * T, np.int32)
    g1, g2 = g.uniform(size=(T, 2)), g.uniform(size=(T, 2))
    np.testing.assert_allclose(F.moe_layer(x, idx, g1 + 2 * g2, ex),
                               F.moe_layer(x, idx, g1, ex) + 2 * F.moe_layer(x, idx, g2, ex),
                               rtol=1e-12, atol=1e-12)


def test_rel_err_rows():
    ref = np.array([[1.0, -2.0], [0.5, 0.25]])
    y = ref + np.array([[0.02, 0.0], [0.0, -0.005]])
    row, fro = F.rel_err_rows(y, ref)
    np.testing.assert_allclose(row, [0.01, 0.01])
    assert fro == pytest.approx(np.hypot(0.02, 0.005) / np.linalg.norm(ref))


def _lora(g, d, w, r):
    return (g.standard_normal((r, d)), g.standard_normal((w, r)), g.standard_normal((r, d)),
            g.standard_normal((w, r)), g.standard_normal((r, w)), g.standard_normal((d, r)))


def test_lora_zero_b_is_base_expert():
    g = np.random.default_rng(5)
    d, w, r = 6, 4, 2
    x = g.standard_normal((3, d))
    ex = _experts(g, 1, d, w)[0]
    a1, b1, a3, b3, a2, b2 = _lora(g, d, w, r)
    z = (a1, 0 * b1, a3, 0 * b3, a2, 0 * b2)
    np.testing.assert_allclose(F.expert_lora(x, *ex, z, 2.0), F.expert(x, *ex), rtol=1e-13)


def test_lora_equals_merged_weights():
    """W x + s B (A x) == (W + s B A) x: the adapter form against merged weights."""
    g = np.random.default_rng(6)
    d, w, r, s = 7, 5, 3, 2.0
    x = g.standard_normal((4, d))
    w1, w3, w2 = _experts(g, 1, d, w)[0]
    a1, b1, a3, b3, a2, b2 = _lora(g, d, w, r)
    merged = (w1 + s * b1 @ a1, w3 + s * b3 @ a3, w2 + s * b2 @ a2)
    np.testing.assert_allclose(F.expert_lora(x, w1, w3, w2, (a1, b1, a3, b3, a2, b2), s),
                               F.expert(x, *merged), rtol=1e-11)
    for t in range(4):  # and against naive loops on the merged weights
        np.testing.assert_allclose(F.expert(x[t:t + 1], *merged)[0], _naive_expert(x[t], *merged),
                                   rtol=1e-11)


def test_lora_in_layer_matches_per_expert_sum():
    g = np.random.default_rng(7)
    E, K, d, w, r, T = 3, 2, 5, 4, 2, 6
    x = g.standard_normal((T, d))
    ex = _experts(g, E, d, w)
    sh = _experts(g, 1, d, w)
    ad = [_lora(g, d, w, r), None, _lora(g, d, w, r)]
    sad = [_lora(g, d, w, r)]
    idx = np.array([[0, 1], [2, 0], [1, 2], [0, 2], [2, 1], [1, 0]], np.int32)
    gate = g.uniform(size=(T, K))
    y = F.moe_layer(x, idx, gate, ex, sh, lora=ad, shared_lora=sad, lora_scale=2.0)
    for t in range(T):
        ref = sum(gate[t, k] * (F.expert(x[t:t + 1], *ex[idx[t, k]]) if ad[idx[t, k]] is None else
                                F.expert_lora(x[t:t + 1], *ex[idx[t, k]], ad[idx[t, k]], 2.0))[0]
                  for k in range(K))
        ref = ref + F.expert_lora(x[t:t + 1], *sh[0], sad[0], 2.0)[0]
        np.testing.assert_allclose(y[t], ref, rtol=1e-11)
