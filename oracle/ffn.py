"""Expert FFN and combine oracle (fp64).

Section 3.1 (Eq. topk): y = sum over active experts i of g_i F_i(x); DeepSeek-V2-Lite's shared
experts process every token and add their outputs to y, un-gated. The paper does not spell out F_i;
both models' experts are SwiGLU MLPs, F(x) = W2 (silu(W1 x) * (W3 x)) with silu(u) = u / (1 + e^-u).
No intermediate rounding: every product and sum is fp64.
"""
from __future__ import annotations

import numpy as np


def silu(u):
    """silu(u) = u * sigmoid(u) = u / (1 + exp(-u))."""
    u = np.asarray(u, np.float64)
    with np.errstate(over="ignore"):
        return u / (1.0 + np.exp(-u))


def expert(x, w1, w3, w2):
    """SwiGLU expert on rows of x: W2 (silu(W1 x) * (W3 x)); x [n, d], W1/W3 [w, d], W2 [d, w]."""
    x = np.asarray(x, np.float64)
    g = x @ np.asarray(w1, np.float64).T
    u = x @ np.asarray(w3, np.float64).T
    return (silu(g) * u) @ np.asarray(w2, np.float64).T


def moe_layer(x, idx, gate, experts, shared=()):
    """y[t] = sum_k gate[t,k] F_{idx[t,k]}(x[t]) + sum_s F^shared_s(x[t]).

    ``experts[e]`` and ``shared[s]`` are (W1, W3, W2) triples; an unused routed expert may be None.
    """
    x = np.asarray(x, np.float64)
    T = x.shape[0]
    K = idx.shape[1]
    y = np.zeros_like(x)
    for k in range(K):
        for e in np.unique(idx[:, k]):
            rows = np.nonzero(idx[:, k] == e)[0]
            w1, w3, w2 = experts[int(e)]
            y[rows] += np.asarray(gate, np.float64)[rows, k, None] * expert(x[rows], w1, w3, w2)
    for w1, w3, w2 in shared:
        y += expert(x, w1, w3, w2)
    assert y.shape[0] == T
    return y


def rel_err_rows(y, ref):
    """Per-token-row error max_j |y_j - ref_j| / max_j |ref_j|, and the Frobenius relative error."""
    y = np.asarray(y, np.float64)
    ref = np.asarray(ref, np.float64)
    den = np.maximum(np.abs(ref).max(axis=1), 1e-30)
    row = np.abs(y - ref).max(axis=1) / den
    fro = np.linalg.norm(y - ref) / max(np.linalg.norm(ref), 1e-30)
    return row, fro
