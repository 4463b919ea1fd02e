"""Routing oracle (fp64): router logits, softmax, Top-K under a mask or a prior, gate weights.

Follows Section 3.1 (Eq. topk), Section 3.2 Stage 1 (Eq. stage1) and "Evaluation and inference"
(Eq. inference). Readings where the paper is silent:

* ties in Top-K go to the lower expert index; the K experts are listed by descending score;
* under a hard mask, experts with m_e = 0 are not eligible at all (p_e * 0 = 0 could otherwise tie
  with an in-set expert whose p underflowed); this equals Top-K(p * m) whenever every p_e > 0;
* gate weights always come from p (full softmax over all E routed experts): Mixtral renormalises
  over the active set, DeepSeek uses p_i as is; no routed scaling factor is applied.

Everything is computed in fp64 from the (already rounded) inputs.
"""
from __future__ import annotations

import numpy as np

MODE_TOPK, MODE_HARD_MASK, MODE_SOFT_PRIOR = 0, 1, 2
GATE_RENORM, GATE_PLAIN = 0, 1


def router_logits(x, w_router):
    """z = W x for each token (Section 3.1): x [T, d], W [E, d] -> z [T, E]."""
    return np.asarray(x, np.float64) @ np.asarray(w_router, np.float64).T


def softmax(z):
    """p = softmax(z) over all E routed experts (Section 3.1), row-wise, max-subtracted."""
    z = np.asarray(z, np.float64)
    e = np.exp(z - z.max(axis=-1, keepdims=True))
    return e / e.sum(axis=-1, keepdims=True)


def scores(p, mode, mask=None, prior=None):
    """The score Top-K ranks by, and which experts are eligible.

    TOPK: s = p (Eq. topk). HARD_MASK: s = p * m, only m_e = 1 eligible (Eq. stage1).
    SOFT_PRIOR: s = p * pi, every expert eligible since pi > 0 (Eq. inference).
    """
    p = np.asarray(p, np.float64)
    eligible = np.ones(p.shape, bool)
    if mode == MODE_TOPK:
        s = p.copy()
    elif mode == MODE_HARD_MASK:
        m = np.asarray(mask).astype(np.float64)
        s = p * m
        eligible = np.broadcast_to(m > 0, p.shape).copy()
    elif mode == MODE_SOFT_PRIOR:
        pi = np.asarray(prior, np.float64)
        if not np.all(pi > 0) or not np.all(np.isfinite(pi)):
            raise ValueError("the prior must be positive and finite (Eq. inference)")
        s = p * pi
    else:
        raise ValueError(f"unknown routing mode {mode}")
    return s, eligible


def top_k(s, eligible, K):
    """Indices of the K eligible experts with the largest s, largest first, ties to the lower index.

    Returns (idx [T, K], order [T, E'] of all eligible experts by the same rule).
    """
    s = np.asarray(s, np.float64)
    T, E = s.shape
    idx = np.empty((T, K), np.int32)
    orders = []
    for t in range(T):
        cand = np.nonzero(eligible[t])[0]
        if len(cand) < K:
            raise ValueError("fewer than K eligible experts (the paper requires K <= E')")
        # primary key: score descending; secondary: expert index ascending
        order = cand[np.lexsort((cand, -s[t, cand]))]
        idx[t] = order[:K]
        orders.append(order)
    return idx, orders


def gates(p, idx, gate_mode):
    """Gate weights of the active experts, from p (Section 3.1 after Eq. topk).

    RENORM (Mixtral): g_i = p_i / sum_{j in A} p_j.  PLAIN (DeepSeek): g_i = p_i.
    """
    p = np.asarray(p, np.float64)
    pa = np.take_along_axis(p, idx.astype(np.int64), axis=1)
    if gate_mode == GATE_RENORM:
        return pa / pa.sum(axis=1, keepdims=True)
    if gate_mode == GATE_PLAIN:
        return pa
    raise ValueError(f"unknown gate mode {gate_mode}")


def route(x, w_router, K, mode, gate_mode, mask=None, prior=None):
    """Full routing of a batch of tokens. Returns a dict with

    idx [T,K] int32, gate [T,K] fp64, z, p, s [T,E],
    gap_k [T]: relative gap (s_K - s_{K+1}) / s_K between the K-th selected and the best
      eligible non-selected expert (inf when no such expert exists),
    gap_in [T]: smallest relative gap between adjacent selected experts (inf when K == 1).
    """
    z = router_logits(x, w_router)
    p = softmax(z)
    s, eligible = scores(p, mode, mask, prior)
    idx, orders = top_k(s, eligible, K)
    g = gates(p, idx, gate_mode)
    T = s.shape[0]
    gap_k = np.full(T, np.inf)
    gap_in = np.full(T, np.inf)
    for t in range(T):
        o = orders[t]
        sk = s[t, o[K - 1]]
        if len(o) > K:
            gap_k[t] = (sk - s[t, o[K]]) / sk if sk > 0 else 0.0
        for k in range(K - 1):
            a, b = s[t, o[k]], s[t, o[k + 1]]
            gap_in[t] = min(gap_in[t], (a - b) / a if a > 0 else 0.0)
    return dict(idx=idx, gate=g, z=z, p=p, s=s, gap_k=gap_k, gap_in=gap_in)
