"""Chained decode-stack oracle (fp64): residual stream, RMSNorm, per-layer masked MoE blocks and the
speculative next-layer routing that drives expert prefetch.

TEST INFRASTRUCTURE ONLY (see the package header).

The models of the paper (Mixtral-8x7B, DeepSeek-V2-Lite; Section 4 and Table 4) alternate attention
and MoE blocks on a residual stream, and each block reads the RMS-normalised stream. The hot path
keeps the MoE blocks only, so one decode step of an L-layer stack is, for every token:

    u_l = RMSNorm_l(x_l) = gamma_l * x_l / sqrt(mean_j(x_l[j]^2) + eps)
    (A_l, g_l) = routing of u_l by layer l's router under its soft prior pi_l   (Eq. inference)
    x_{l+1} = x_l + sum_k g_{l,k} F_{A_{l,k}}(u_l) + shared experts(u_l)        (Eq. topk)

Readings (the paper states none of this):
* RMSNorm as the two architectures define it: mean of squares over the d hidden units, eps inside
  the square root (1e-5 for Mixtral, 1e-6 for DeepSeek-V2-Lite), a learned per-unit scale gamma.
* Prefetch prediction (offloading systems load experts ahead of need, Section 2 "Offloading
  systems for MoE inference"; the paper gives no rule of its own): while layer l runs, layer
  l+1's experts are predicted by routing RMSNorm_{l+1}(x_l), i.e. layer l+1's norm,
  router and prior applied to the stream before layer l adds its output. The prefetch candidates
  of a step are the distinct predicted experts ranked by how many (token, k) predictions name them,
  then by the best rank k at which any token predicts them (the K predictions of a token are in
  descending score), then by id; the cache loads at most n_max of them (oracle.cache).
"""
from __future__ import annotations

import numpy as np

from . import ffn as F
from . import routing as R


def rmsnorm(x, gamma, eps):
    """gamma * x / sqrt(mean(x^2) + eps) for each row of x [T, d] (fp64)."""
    x = np.asarray(x, np.float64)
    ms = np.mean(x * x, axis=-1, keepdims=True)
    return np.asarray(gamma, np.float64) * x / np.sqrt(ms + eps)


def route_layer(u, layer, K, gate_mode):
    """Soft-prior routing of normalised inputs u by one layer (Eq. inference)."""
    return R.route(u, layer["router"], K, R.MODE_SOFT_PRIOR, gate_mode, prior=layer["prior"])


def chain(x0, layers, K, gate_mode, eps, predict=False):
    """One decode step of the stack for the tokens x0 [T, d].

    layers[l] is a dict with router [E, d], prior [E], gamma [d], experts (E (W1, W3, W2) triples,
    None where unused) and shared (list of triples). Returns (x_L, per-layer records), each record
    holding x (the stream entering the layer), u, the routing dict r, y (the block output) and,
    with predict=True and a next layer, pred = the routing of RMSNorm_{l+1}(x_l) by layer l+1.
    """
    x = np.asarray(x0, np.float64)
    recs = []
    for l, ly in enumerate(layers):
        u = rmsnorm(x, ly["gamma"], eps)
        r = route_layer(u, ly, K, gate_mode)
        y = F.moe_layer(u, r["idx"], r["gate"], ly["experts"], ly.get("shared", ()))
        rec = dict(x=x, u=u, r=r, y=y)
        if predict and l + 1 < len(layers):
            nxt = layers[l + 1]
            rec["pred"] = route_layer(rmsnorm(x, nxt["gamma"], eps), nxt, K, gate_mode)
        recs.append(rec)
        x = x + y
    return x, recs


def prefetch_candidates(idx_pred):
    """Prefetch candidates from predicted routing idx_pred [T, K] (each row in descending score):
    distinct ids ranked by the number of predictions naming them (descending), then the best rank
    k at which they are predicted (ascending), then id (ascending)."""
    idx_pred = np.asarray(idx_pred)
    count, best = {}, {}
    for row in idx_pred:
        for k, e in enumerate(row.tolist()):
            count[e] = count.get(e, 0) + 1
            best[e] = min(best.get(e, k), k)
    ranked = sorted(count, key=lambda e: (-count[e], best[e], e))
    return [int(e) for e in ranked]
