"""Stage-1 mask machinery oracle (fp64): mask sampling and the straight-through mask gradient.

Section 3.2 "Stage 1" (Eq. stage1): pi = softmax(m~); m = MultinomialSample(pi, E'), E' distinct
experts drawn without replacement; A = TopK(p * m); gates computed from p * m.
Section 3.2 "Mask optimization" (Eq. ste): the loss reaches m through the gate weights of the
active experts, dL/dm sums every token's contribution, the straight-through estimator passes it
to pi, and the softmax Jacobian carries it to m~: dL/dm~ = (diag(pi) - pi pi^T) dL/dm.

Readings:
* MultinomialSample is realised by the Gumbel-top-k rule: with one uniform u_e per expert,
  key_e = log(pi_e) - log(-log(u_e)) and the E' largest keys are drawn (ties to the lower index).
  This has the law of E' sequential draws without replacement (Gumbel-max trick applied
  repeatedly); the pins check that law. The uniforms are inputs (drawn by the caller).
* Gates from p * m, with m_e = 1 on A: Mixtral renormalises, g_i = p_i m_i / sum_{j in A} p_j m_j,
  so dg_i/dm_k = delta_ik g_i - g_i g_k for k in A; DeepSeek uses g_i = p_i m_i, so
  dg_i/dm_k = delta_ik g_i. Experts outside A_t receive nothing from token t (Top-K selection is
  piecewise constant in m).
* dL/dg_{t,k} = < dL/dy_t , F_{A_{t,k}}(x_t) > since y_t = sum_k g_{t,k} F_{A_{t,k}}(x_t) + shared.
"""
from __future__ import annotations

import numpy as np

GATE_RENORM, GATE_PLAIN = 0, 1


def softmax(v):
    v = np.asarray(v, np.float64)
    e = np.exp(v - v.max(axis=-1, keepdims=True))
    return e / e.sum(axis=-1, keepdims=True)


def sample_mask(m_tilde, uniforms, e_keep):
    """Binary masks [L, E] with e_keep ones: the Gumbel-top-k draw from pi = softmax(m~) with the
    given uniforms in (0, 1). Returns (mask, pi, keys)."""
    m_tilde = np.atleast_2d(np.asarray(m_tilde, np.float64))
    u = np.atleast_2d(np.asarray(uniforms, np.float64))
    pi = softmax(m_tilde)
    keys = np.log(pi) - np.log(-np.log(u))
    L, E = pi.shape
    mask = np.zeros((L, E), np.uint8)
    for l in range(L):
        order = np.lexsort((np.arange(E), -keys[l]))  # key descending, index ascending
        mask[l, order[:e_keep]] = 1
    return mask, pi, keys


def sequential_set_probabilities(pi, e_keep):
    """Exact law of the SET drawn by e_keep sequential draws without replacement from pi
    (enumeration over ordered draws; small E only). Returns {frozenset: probability}."""
    import itertools

    pi = np.asarray(pi, np.float64)
    E = len(pi)
    out = {}
    for seq in itertools.permutations(range(E), e_keep):
        p, left = 1.0, 1.0
        for e in seq:
            p *= pi[e] / left
            left -= pi[e]
        key = frozenset(seq)
        out[key] = out.get(key, 0.0) + p
    return out


def gate_grad(dy, expert_out):
    """dL/dg_{t,k} = < dL/dy_t , F_{A_{t,k}}(x_t) >: dy [T, d], expert_out [T, K, d]."""
    return np.einsum("td,tkd->tk", np.asarray(dy, np.float64), np.asarray(expert_out, np.float64))


def mask_grad(idx, gate, dgate, gate_mode, E):
    """dL/dm [E] summed over tokens (Eq. ste, through the gates of the active experts)."""
    idx = np.asarray(idx)
    g = np.asarray(gate, np.float64)
    dg = np.asarray(dgate, np.float64)
    dm = np.zeros(E)
    T, K = idx.shape
    for t in range(T):
        inner = float(np.dot(g[t], dg[t]))  # sum_{i in A} g_i dL/dg_i
        for k in range(K):
            e = int(idx[t, k])
            if gate_mode == GATE_RENORM:
                dm[e] += g[t, k] * (dg[t, k] - inner)
            else:
                dm[e] += g[t, k] * dg[t, k]
    return dm


def mask_tilde_grad(pi, dm):
    """dL/dm~ = (diag(pi) - pi pi^T) dL/dm (straight-through, then the softmax Jacobian)."""
    pi = np.asarray(pi, np.float64)
    return (np.diag(pi) - np.outer(pi, pi)) @ np.asarray(dm, np.float64)


def gates_from_masked(p, active, m, gate_mode):
    """Gates of the active experts computed from p * m with a real-valued m (for the pins)."""
    p = np.asarray(p, np.float64)
    pm = p[active] * np.asarray(m, np.float64)[active]
    return pm / pm.sum() if gate_mode == GATE_RENORM else pm
