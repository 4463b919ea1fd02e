"""Pins of the Stage-1 mask oracle (Section 3.2 Eq. stage1 and Eq. ste).

The sampler against the exact law of sequential draws without replacement (enumeration on tiny
E, frequencies over many draws); the mask gradient against finite differences of the gate
function of p * m; the softmax Jacobian against finite differences of softmax; the gate gradient
against finite differences of the layer output."""
import numpy as np
import pytest

from oracle import ffn as F
from oracle import mask as Mk


def test_sampler_draws_exactly_e_keep_distinct_experts():
    g = np.random.default_rng(0)
    m_t = g.standard_normal((5, 16))
    u = g.uniform(size=(5, 16))
    mask, pi, keys = Mk.sample_mask(m_t, u, 12)
    assert np.all(mask.sum(axis=1) == 12)
    np.testing.assert_allclose(pi.sum(axis=1), 1.0)
    # the drawn experts are exactly those with the 12 largest keys
    for l in range(5):
        assert set(np.nonzero(mask[l])[0]) == set(np.argsort(-keys[l])[:12])


@pytest.mark.parametrize("e_keep", [1, 2, 3])
def test_sampler_law_equals_sequential_draws(e_keep):
    """Frequencies of the drawn SET over 200k Gumbel-top-k draws match the exact probabilities of
    sequential multinomial draws without replacement (within 5 standard errors)."""
    E, N = 5, 200_000
    m_t = np.array([0.3, -1.0, 1.2, 0.0, 0.7])
    g = np.random.default_rng(1 + e_keep)
    mask, pi, _ = Mk.sample_mask(np.tile(m_t, (N, 1)), g.uniform(size=(N, E)), e_keep)
    exact = Mk.sequential_set_probabilities(pi[0], e_keep)
    counts = {}
    for row in mask:
        key = frozenset(np.nonzero(row)[0].tolist())
        counts[key] = counts.get(key, 0) + 1
    assert set(counts) <= set(exact)
    for key, p in exact.items():
        f = counts.get(key, 0) / N
        assert abs(f - p) <= 5 * np.sqrt(p * (1 - p) / N) + 1e-4, (key, f, p)


def test_uniform_prior_first_draw_is_uniform():
    E, N = 8, 100_000
    mask, _, _ = Mk.sample_mask(np.zeros((N, E)), np.random.default_rng(2).uniform(size=(N, E)), 1)
    freq = mask.mean(axis=0)
    np.testing.assert_allclose(freq, 1 / E, atol=5 * np.sqrt((1 / E) * (1 - 1 / E) / N))


@pytest.mark.parametrize("gate_mode", [Mk.GATE_RENORM, Mk.GATE_PLAIN])
def test_mask_grad_matches_finite_differences(gate_mode):
    """L = sum_t sum_k dgate_{t,k} g_{t,k}(m): dL/dm_e from the oracle equals a central difference
    of the gates computed from p * m around m = 1."""
    g = np.random.default_rng(3)
    T, E, K = 6, 8, 3
    p = np.stack([Mk.softmax(g.standard_normal(E) * 2) for _ in range(T)])
    idx = np.stack([g.permutation(E)[:K] for _ in range(T)]).astype(np.int32)
    gate = np.stack([Mk.gates_from_masked(p[t], idx[t], np.ones(E), gate_mode) for t in range(T)])
    dgate = g.standard_normal((T, K))
    dm = Mk.mask_grad(idx, gate, dgate, gate_mode, E)

    def loss(m):
        return sum(float(np.dot(dgate[t], Mk.gates_from_masked(p[t], idx[t], m, gate_mode)))
                   for t in range(T))

    eps = 1e-6
    for e in range(E):
        mp, mm = np.ones(E), np.ones(E)
        mp[e] += eps
        mm[e] -= eps
        assert dm[e] == pytest.approx((loss(mp) - loss(mm)) / (2 * eps), rel=1e-6, abs=1e-8)


def test_softmax_jacobian_and_zero_sum():
    g = np.random.default_rng(4)
    m_t = g.standard_normal(8)
    pi = Mk.softmax(m_t)
    dm = g.standard_normal(8)
    dmt = Mk.mask_tilde_grad(pi, dm)
    eps = 1e-6
    for j in range(8):
        a, b = m_t.copy(), m_t.copy()
        a[j] += eps
        b[j] -= eps
        # d/dm~_j of <dm, softmax(m~)> (the straight-through chain)
        fd = (np.dot(dm, Mk.softmax(a)) - np.dot(dm, Mk.softmax(b))) / (2 * eps)
        assert dmt[j] == pytest.approx(fd, rel=1e-6, abs=1e-9)
    assert abs(dmt.sum()) < 1e-12  # rows of diag(pi) - pi pi^T sum to zero


def test_gate_grad_matches_layer_finite_differences():
    g = np.random.default_rng(5)
    T, E, K, d, w = 3, 4, 2, 6, 5
    x = g.standard_normal((T, d))
    ex = [(g.standard_normal((w, d)), g.standard_normal((w, d)), g.standard_normal((d, w)))
          for _ in range(E)]
    idx = np.array([[0, 2], [1, 3], [2, 0]], np.int32)
    gate = g.uniform(size=(T, K))
    dy = g.standard_normal((T, d))
    outs = np.stack([np.stack([F.expert(x[t:t + 1], *ex[idx[t, k]])[0] for k in range(K)])
                     for t in range(T)])
    dg = Mk.gate_grad(dy, outs)
    eps = 1e-6
    for t in range(T):
        for k in range(K):
            a, b = gate.copy(), gate.copy()
            a[t, k] += eps
            b[t, k] -= eps
            fd = (np.sum(dy * F.moe_layer(x, idx, a, ex)) - np.sum(dy * F.moe_layer(x, idx, b, ex))) / (2 * eps)
            assert dg[t, k] == pytest.approx(fd, rel=1e-6)
