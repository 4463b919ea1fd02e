"""Pins of the routing oracle (Section 3.1 Eq. topk, Section 3.2 Eq. stage1, Eq. inference).

Each test ties the oracle to something other than itself: brute force over all subsets, closed
forms of the gates in terms of the logits, a library softmax, naive loops, and the properties the
paper states (a hard mask never selects a masked expert; a positive prior excludes no expert; gates
in the masked stage equal the unmasked ones on the active set).
"""
import itertools

import numpy as np
import pytest
import scipy.special

from oracle import routing as R


def _rand(seed, T, E, d, scale=1.0):
    g = np.random.default_rng(seed)
    return g.standard_normal((T, d)) * scale, g.standard_normal((E, d)) * 0.02 * scale


def test_router_logits_naive_loop():
    x, w = _rand(0, 3, 5, 7)
    z = R.router_logits(x, w)
    for t in range(3):
        for e in range(5):
            acc = 0.0
            for j in range(7):
                acc += x[t, j] * w[e, j]
            assert z[t, e] == pytest.approx(acc, rel=1e-13, abs=1e-15)


def test_softmax_matches_library():
    z = np.random.default_rng(1).standard_normal((11, 64)) * 5
    np.testing.assert_allclose(R.softmax(z), scipy.special.softmax(z, axis=1), rtol=1e-13)
    # shift invariance and extreme logits stay finite
    np.testing.assert_allclose(R.softmax(z + 1000.0), R.softmax(z), rtol=1e-12)


def _brute_force_topk(s, eligible, K):
    """All K-subsets of the eligible experts; the Top-K set is the unique subset whose smallest
    key beats the largest key outside it, key = (score, -index)."""
    E = len(s)
    cand = [e for e in range(E) if eligible[e]]
    key = lambda e: (s[e], -e)
    found = []
    for sub in itertools.combinations(cand, K):
        rest = [e for e in cand if e not in sub]
        if not rest or min(key(e) for e in sub) > max(key(e) for e in rest):
            found.append(sub)
    assert len(found) == 1
    return sorted(found[0], key=lambda e: (-s[e], e))


@pytest.mark.parametrize("mode", [R.MODE_TOPK, R.MODE_HARD_MASK, R.MODE_SOFT_PRIOR])
@pytest.mark.parametrize("E,K", [(4, 1), (6, 2), (8, 2), (8, 3), (8, 8)])
def test_topk_brute_force(mode, E, K):
    g = np.random.default_rng(E * 10 + K + mode)
    x, w = _rand(E + K, 40, E, 16, scale=3.0)
    mask = np.zeros(E, np.uint8)
    mask[g.permutation(E)[: max(K, E // 2 + 1)]] = 1
    prior = g.uniform(0.01, 1.0, E)
    if mode == R.MODE_HARD_MASK and K == E:
        mask[:] = 1
    out = R.route(x, w, K, mode, R.GATE_RENORM, mask=mask, prior=prior)
    for t in range(40):
        s = out["s"][t]
        elig = np.ones(E, bool) if mode != R.MODE_HARD_MASK else mask > 0
        assert list(out["idx"][t]) == _brute_force_topk(s, elig, K)


def test_exact_ties_go_to_lower_index():
    # x = 0 gives z = 0 for every expert: all scores tie exactly
    x = np.zeros((2, 8))
    w = np.random.default_rng(2).standard_normal((8, 8))
    out = R.route(x, w, 3, R.MODE_TOPK, R.GATE_RENORM)
    assert out["idx"].tolist() == [[0, 1, 2], [0, 1, 2]]
    out = R.route(x, w, 2, R.MODE_HARD_MASK, R.GATE_RENORM, mask=np.array([0, 0, 1, 0, 1, 1, 0, 0]))
    assert out["idx"].tolist() == [[2, 4], [2, 4]]
    np.testing.assert_allclose(out["gate"], 0.5)


def test_all_ones_mask_is_plain_topk():
    x, w = _rand(3, 200, 8, 32, scale=2.0)
    plain = R.route(x, w, 2, R.MODE_TOPK, R.GATE_RENORM)
    masked = R.route(x, w, 2, R.MODE_HARD_MASK, R.GATE_RENORM, mask=np.ones(8, np.uint8))
    assert np.array_equal(plain["idx"], masked["idx"])
    assert np.array_equal(plain["gate"], masked["gate"])


@pytest.mark.parametrize("E", [8, 64])
def test_uniform_prior_is_plain_topk_bit_exact(E):
    # pi = 1/E with E a power of two: p * pi is an exact scaling, so the ranking is unchanged
    x, w = _rand(4, 300, E, 32, scale=2.0)
    K = 6 if E == 64 else 2
    plain = R.route(x, w, K, R.MODE_TOPK, R.GATE_PLAIN)
    soft = R.route(x, w, K, R.MODE_SOFT_PRIOR, R.GATE_PLAIN, prior=np.full(E, 1.0 / E))
    assert np.array_equal(plain["idx"], soft["idx"])
    assert np.array_equal(plain["gate"], soft["gate"])


def test_hard_mask_never_selects_masked_expert():
    E, K = 64, 6
    x, w = _rand(5, 500, E, 64, scale=3.0)
    mask = np.zeros(E, np.uint8)
    mask[np.random.default_rng(5).permutation(E)[:16]] = 1
    out = R.route(x, w, K, R.MODE_HARD_MASK, R.GATE_PLAIN, mask=mask)
    assert np.all(mask[out["idx"]] == 1)


def test_soft_prior_keeps_every_expert_selectable():
    # For each expert outside the kept set: a token aligned with its router row selects it anyway
    E, K, d = 8, 2, 64
    g = np.random.default_rng(6)
    w = g.standard_normal((E, d)) * 0.02
    mask = np.array([1, 1, 1, 1, 0, 0, 0, 0], np.uint8)
    prior = np.exp(2.0 * mask) / np.exp(2.0 * mask).sum()
    for e in range(4, 8):
        x = 400.0 * w[e][None, :]
        out = R.route(x, w, K, R.MODE_SOFT_PRIOR, R.GATE_RENORM, prior=prior)
        assert e in out["idx"][0]
        # closed form: e is chosen iff z_e + log pi_e beats the K-th best of the others
        z = out["z"][0]
        b = z + np.log(prior)
        others = np.sort(np.delete(b, e))[::-1]
        assert b[e] > others[K - 1]
    # while a hard mask with the same set never can
    out = R.route(400.0 * w[5][None, :], w, K, R.MODE_HARD_MASK, R.GATE_RENORM, mask=mask)
    assert 5 not in out["idx"][0]


def test_soft_prior_ranking_equals_log_domain_ranking():
    # p_e pi_e is ranked like z_e + log pi_e (log is monotone; softmax shares one denominator)
    E, K = 64, 6
    x, w = _rand(7, 200, E, 128, scale=2.0)
    prior = np.random.default_rng(7).uniform(0.001, 0.1, E)
    out = R.route(x, w, K, R.MODE_SOFT_PRIOR, R.GATE_PLAIN, prior=prior)
    b = out["z"] + np.log(prior)[None, :]
    for t in range(200):
        if out["gap_k"][t] < 1e-9 or out["gap_in"][t] < 1e-9:
            continue
        assert list(out["idx"][t]) == list(np.argsort(-b[t], kind="stable")[:K])


def test_gate_closed_forms():
    E, K = 8, 2
    x, w = _rand(8, 100, E, 32, scale=2.0)
    mask = np.array([0, 1, 1, 0, 1, 0, 1, 0], np.uint8)
    prior = np.random.default_rng(8).uniform(0.05, 0.5, E)
    for mode in (R.MODE_TOPK, R.MODE_HARD_MASK, R.MODE_SOFT_PRIOR):
        ren = R.route(x, w, K, mode, R.GATE_RENORM, mask=mask, prior=prior)
        pla = R.route(x, w, K, mode, R.GATE_PLAIN, mask=mask, prior=prior)
        z = ren["z"]
        for t in range(100):
            a = ren["idx"][t]
            # RENORM: exp(z_i) / sum_{j in A} exp(z_j); PLAIN: exp(z_i) / sum_all exp(z_j)
            ea = np.exp(z[t, a])
            np.testing.assert_allclose(ren["gate"][t], ea / ea.sum(), rtol=1e-12)
            np.testing.assert_allclose(pla["gate"][t], ea / np.exp(z[t]).sum(), rtol=1e-12)
        np.testing.assert_allclose(ren["gate"].sum(axis=1), 1.0, rtol=1e-12)


def test_hard_mask_gates_equal_unmasked_gates_on_active_set():
    # Section 3.2: on A, gates from p * m equal gates from p since m_i = 1 there
    E, K = 8, 2
    x, w = _rand(9, 100, E, 32, scale=2.0)
    mask = np.array([1, 0, 1, 1, 0, 1, 0, 0], np.uint8)
    out = R.route(x, w, K, R.MODE_HARD_MASK, R.GATE_PLAIN, mask=mask)
    pm = out["p"] * mask[None, :]
    np.testing.assert_allclose(out["gate"], np.take_along_axis(pm, out["idx"].astype(int), 1),
                               rtol=1e-15)


def test_gaps_flag_near_ties():
    x = np.array([[1.0, 0.0], [1.0, 1e-6]])
    w = np.array([[1.0, 0.0], [1.0, 0.0], [0.0, 1.0]])
    out = R.route(x, w, 1, R.MODE_TOPK, R.GATE_RENORM)
    # token 0: experts 0 and 1 tie exactly -> gap 0; token 1: the same
    assert out["gap_k"][0] == 0.0 and out["gap_k"][1] == 0.0
    assert out["idx"][:, 0].tolist() == [0, 0]


def test_invalid_inputs_rejected():
    x, w = _rand(10, 2, 4, 8)
    with pytest.raises(ValueError):
        R.route(x, w, 2, R.MODE_HARD_MASK, R.GATE_RENORM, mask=np.array([1, 0, 0, 0]))
    with pytest.raises(ValueError):
        R.route(x, w, 2, R.MODE_SOFT_PRIOR, R.GATE_RENORM, prior=np.array([0.5, 0.5, 0.0, 0.1]))
