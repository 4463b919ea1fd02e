"""Expert FFN and combine oracle (fp64).

Section 3.1 (Eq. topk): y = sum over active experts i of g_i F_i(x); DeepSeek-V2-Lite's shared
experts process every token and add their outputs to y, un-gated. The paper does not spell out F_i;
both models' experts are SwiGLU MLPs, F(x) = W2 (silu(W1 x) * (W3 x)) with silu(u) = u / (1 + e^-u).
In Stage 2 (Section 3.2; rank 8, alpha 16 in Appendix B) the experts carry LoRA adapters: each
projection W becomes W x + (alpha / r) B (A x); the adapters are applied to W1, W3 and W2 (reading:
"all routed experts ... with LoRA" adapts every linear map of an expert; no dropout in a forward
whose result is compared). No intermediate rounding: every product and sum is fp64.
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


def lora_linear(x, w, a, b, scale):
    """LoRA-adapted projection (Stage 2 fine-tunes the experts with LoRA, Section 3.2):
    W x + scale * B (A x), with A [r, in], B [out, r], scale = alpha / r; x holds rows."""
    x = np.asarray(x, np.float64)
    base = x @ np.asarray(w, np.float64).T
    if a is None:
        return base
    return base + scale * ((x @ np.asarray(a, np.float64).T) @ np.asarray(b, np.float64).T)


def expert_lora(x, w1, w3, w2, lora, scale):
    """SwiGLU expert whose three projections carry LoRA adapters:
    lora = (A1, B1, A3, B3, A2, B2) for W1 (gate), W3 (up) and W2 (down)."""
    a1, b1, a3, b3, a2, b2 = lora
    g = lora_linear(x, w1, a1, b1, scale)
    u = lora_linear(x, w3, a3, b3, scale)
    return lora_linear(silu(g) * u, w2, a2, b2, scale)


def moe_layer(x, idx, gate, experts, shared=(), lora=None, shared_lora=None, lora_scale=0.0):
    """y[t] = sum_k gate[t,k] F_{idx[t,k]}(x[t]) + sum_s F^shared_s(x[t]).

    ``experts[e]`` and ``shared[s]`` are (W1, W3, W2) triples; an unused routed expert may be None.
    ``lora[e]`` / ``shared_lora[s]``, when given, are (A1, B1, A3, B3, A2, B2) adapters (or None)
    applied with ``lora_scale`` = alpha / r.
    """
    x = np.asarray(x, np.float64)
    T = x.shape[0]
    K = idx.shape[1]
    y = np.zeros_like(x)

    def F(rows_x, ex, ad):
        return expert(rows_x, *ex) if ad is None else expert_lora(rows_x, *ex, ad, lora_scale)

    for k in range(K):
        for e in np.unique(idx[:, k]):
            rows = np.nonzero(idx[:, k] == e)[0]
            ad = None if lora is None else lora[int(e)]
            y[rows] += np.asarray(gate, np.float64)[rows, k, None] * F(x[rows], experts[int(e)], ad)
    for s, ex in enumerate(shared):
        ad = None if shared_lora is None else shared_lora[s]
        y += F(x, ex, ad)
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
