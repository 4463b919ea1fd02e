"""Pins of the chained-stack oracle: RMSNorm, the residual chain and the prefetch prediction.

RMSNorm against its defining invariants (unit RMS, scale invariance, a closed form for a constant
row, the per-unit scale); the chain against symmetries of its definition (scaling the stream and
every down projection scales every residual and leaves every routing unchanged; zero down
projections leave the stream unchanged, so the prediction for layer l+1 is exact) and against a
closed form for identity-like experts written with math.exp elementwise; the prefetch set against
hand-worked rankings."""
import math

import numpy as np
import pytest

from oracle import routing as R
from oracle import stack as S


def test_rmsnorm_unit_rms_and_scale_invariance():
    g = np.random.default_rng(0)
    x = g.standard_normal((5, 64)) * g.uniform(0.1, 10, size=(5, 1))
    u = S.rmsnorm(x, np.ones(64), 0.0)
    np.testing.assert_allclose(np.sqrt(np.mean(u * u, axis=1)), 1.0, rtol=1e-14)
    for c in (1e-3, 0.5, 7.0, 1e4):
        np.testing.assert_allclose(S.rmsnorm(c * x, np.ones(64), 0.0), u, rtol=1e-13)
    gamma = g.uniform(0.5, 1.5, 64)
    np.testing.assert_allclose(S.rmsnorm(x, gamma, 0.0), gamma * u, rtol=1e-14)


def test_rmsnorm_constant_row_closed_form():
    """A row of d copies of c: mean square c^2, so every unit is c / sqrt(c^2 + eps)."""
    for c in (-3.0, 0.01, 2.5):
        for eps in (0.0, 1e-6, 1e-5, 0.1):
            u = S.rmsnorm(np.full((1, 32), c), np.ones(32), eps)
            np.testing.assert_allclose(u, c / math.sqrt(c * c + eps), rtol=1e-15)
    np.testing.assert_array_equal(S.rmsnorm(np.zeros((1, 8)), np.ones(8), 1e-5), 0.0)


def _layers(g, L, E, d, w, gamma_spread=0.3, zero_w2=()):
    layers = []
    for l in range(L):
        experts = []
        for _ in range(E):
            w2 = np.zeros((d, w)) if l in zero_w2 else g.standard_normal((d, w)) * 0.3
            experts.append((g.standard_normal((w, d)) * 0.3, g.standard_normal((w, d)) * 0.3, w2))
        prior = g.uniform(0.2, 1.0, E)
        layers.append(dict(router=g.standard_normal((E, d)), prior=prior / prior.sum(),
                           gamma=1.0 + gamma_spread * g.standard_normal(d), experts=experts))
    return layers


def test_chain_scales_with_the_stream():
    """x0 -> c x0 and every W2 -> c W2: every u_l is unchanged (RMSNorm, eps = 0), so every routing
    is unchanged and every x_l scales by c. Fails if the residual adds u instead of x, if the
    norm is dropped or applied to y, or if a layer reads x0 instead of x_l."""
    g = np.random.default_rng(1)
    L, E, K, d, w, T = 4, 6, 2, 12, 10, 7
    layers = _layers(g, L, E, d, w)
    x0 = g.standard_normal((T, d))
    c = 3.7
    scaled = [dict(ly, experts=[(a, b, c * w2) for a, b, w2 in ly["experts"]]) for ly in layers]
    xa, ra = S.chain(x0, layers, K, R.GATE_RENORM, 0.0)
    xb, rb = S.chain(c * x0, scaled, K, R.GATE_RENORM, 0.0)
    np.testing.assert_allclose(xb, c * xa, rtol=1e-12, atol=1e-12)
    for a, b in zip(ra, rb):
        np.testing.assert_array_equal(a["r"]["idx"], b["r"]["idx"])
        np.testing.assert_allclose(b["x"], c * a["x"], rtol=1e-12, atol=1e-12)
    # and the chain really moves the stream (the symmetry is not vacuous)
    assert np.abs(xa - x0).max() > 1.0


def test_zero_down_projections_leave_the_stream_and_make_prediction_exact():
    g = np.random.default_rng(2)
    L, E, K, d, w, T = 5, 8, 3, 16, 8, 9
    layers = _layers(g, L, E, d, w, zero_w2=range(L))
    x0 = g.standard_normal((T, d))
    xL, recs = S.chain(x0, layers, K, R.GATE_PLAIN, 1e-6, predict=True)
    np.testing.assert_array_equal(xL, x0)
    for l in range(L - 1):
        np.testing.assert_array_equal(recs[l]["pred"]["idx"], recs[l + 1]["r"]["idx"])
    # per-layer norm scales differ, so the layers route differently (the check above is not vacuous)
    assert any(not np.array_equal(recs[0]["r"]["idx"], r["r"]["idx"]) for r in recs[1:])


def test_identity_experts_closed_form():
    """E = 2 identical experts with W1 = W3 = a I and W2 = I (d = w), K = 1, renormalised gate 1:
    x1 = x0 + silu(a u) a u elementwise with u = RMSNorm(x0), silu(v) = v / (1 + e^-v)."""
    g = np.random.default_rng(3)
    d, T, a, eps = 8, 4, 0.7, 1e-5
    I = np.eye(d)
    gamma = 1.0 + 0.2 * g.standard_normal(d)
    ex = (a * I, a * I, I)
    layer = dict(router=g.standard_normal((2, d)), prior=np.array([0.5, 0.5]), gamma=gamma,
                 experts=[ex, ex])
    x0 = g.standard_normal((T, d))
    x1, _ = S.chain(x0, [layer], 1, R.GATE_RENORM, eps)
    for t in range(T):
        ms = sum(v * v for v in x0[t]) / d
        for j in range(d):
            u = gamma[j] * x0[t, j] / math.sqrt(ms + eps)
            v = a * u
            assert x1[t, j] == pytest.approx(x0[t, j] + v / (1.0 + math.exp(-v)) * v, rel=1e-12, abs=1e-14)


def test_prefetch_candidate_ranking():
    """Hand-worked: counts first, then the best predicted rank, then the id."""
    assert S.prefetch_candidates(np.array([[3, 1], [1, 2], [2, 1]])) == [1, 2, 3]
    assert S.prefetch_candidates(np.array([[5, 0], [0, 5]])) == [0, 5]   # same count, both rank 0
    assert S.prefetch_candidates(np.array([[7, 2, 4]])) == [7, 2, 4]     # one token: its own order
    assert S.prefetch_candidates(np.array([[4, 1], [1, 3]])) == [1, 4, 3]  # 4 at rank 0, 3 at 1
    assert S.prefetch_candidates(np.array([[6, 3], [2, 6]])) == [6, 2, 3]  # 2 at rank 0 beats 3
