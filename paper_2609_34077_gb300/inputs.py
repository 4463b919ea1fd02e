"""Seeded synthetic inputs for the masked MoE layer (hidden states, weights, masks, priors).

This module holds no step of the method: it only draws random numbers and shapes them into the
tensors a caller passes in. Both the CUDA path and the CPU oracle receive the same arrays from here.

Recipe (all draws are Philox4x32-10 counter-based streams from numpy, keyed by
``(seed, tensor id, chunk)``, so the values do not depend on thread count or machine):

* weights (router, W1, W3, W2 of every expert): N(0, 0.02^2), drawn in fp32 and rounded to bf16
  (round-to-nearest-even) for the bf16 shapes; kept fp32 for the tiny fp32 shape;
* prefill hidden states: i.i.d. N(0, 1);
* decode hidden states: one AR(1) stream per (layer, batch row),
  ``x_0 = e_0 / sqrt(1 - rho^2)`` (stationary start), ``x_t = rho x_{t-1} + e_t``, ``e_t ~ N(0, 1)``,
  rho = 0.8, generated in fp32 then rounded to bf16;
* keep-k masks: a seeded Fisher-Yates shuffle of the E expert ids, first k ids kept;
* soft-prior stand-in for the learned mask: ``m~ = gamma * m`` with gamma = 2, and
  ``pi = softmax(m~)`` (the map the paper's Stage 1 uses to turn m~ into pi);
* RMSNorm scales of a chained stack: ``1 + N(0, 0.1^2)`` per hidden unit, per layer; the stream
  entering the stack: the AR(1) recipe above, kept in fp32 (the residual stream's precision).
"""
from __future__ import annotations

import hashlib
import math
from concurrent.futures import ThreadPoolExecutor
from dataclasses import dataclass, field

import numpy as np
import torch

ROUTE_TOPK, ROUTE_HARD_MASK, ROUTE_SOFT_PRIOR = 0, 1, 2
GATE_RENORM, GATE_PLAIN = 0, 1
F32, BF16 = 0, 1

_CHUNK = 1 << 22
_POOL = ThreadPoolExecutor(max_workers=16)


@dataclass(frozen=True)
class LayerShape:
    """Shape of one MoE layer: hidden d, E routed experts, top-K, SwiGLU width w, S shared experts."""
    name: str
    d: int
    E: int
    K: int
    w: int
    n_shared: int
    gate: int
    dtype: int
    cache_slots: int
    keep: int  # experts kept by the stand-in mask
    norm_eps: float = 1e-5  # RMSNorm epsilon of the model's block inputs

    @property
    def expert_elems(self) -> int:
        """Elements of one packed expert block [W1 (w x d) | W3 (w x d) | W2 (d x w)]."""
        return 3 * self.w * self.d

    @property
    def expert_bytes(self) -> int:
        return self.expert_elems * (2 if self.dtype == BF16 else 4)


TINY = LayerShape("tiny-fp32", d=256, E=8, K=2, w=512, n_shared=0, gate=GATE_RENORM, dtype=F32,
                  cache_slots=4, keep=4)
MIXTRAL = LayerShape("mixtral-8x7b", d=4096, E=8, K=2, w=14336, n_shared=0, gate=GATE_RENORM,
                     dtype=BF16, cache_slots=4, keep=4)
DSV2_LITE = LayerShape("deepseek-v2-lite", d=2048, E=64, K=6, w=1408, n_shared=2, gate=GATE_PLAIN,
                       dtype=BF16, cache_slots=12, keep=16, norm_eps=1e-6)


def _key(seed: int, *ids) -> int:
    h = hashlib.sha256(repr((seed,) + tuple(ids)).encode()).digest()
    return int.from_bytes(h[:16], "little")


def normal_f32(seed: int, tensor_id, n: int, std: float = 1.0) -> np.ndarray:
    """n draws of N(0, std^2) in fp32 from Philox keyed by (seed, tensor_id, chunk)."""
    out = np.empty(n, np.float32)

    def fill(c):
        s = c * _CHUNK
        e = min(n, s + _CHUNK)
        g = np.random.Generator(np.random.Philox(key=_key(seed, tensor_id, c)))
        g.standard_normal(out=out[s:e], dtype=np.float32)

    list(_POOL.map(fill, range((n + _CHUNK - 1) // _CHUNK)))
    if std != 1.0:
        out *= np.float32(std)
    return out


def as_dtype(a: np.ndarray, dtype: int) -> torch.Tensor:
    """fp32 array -> CPU tensor of the layer dtype (bf16 rounding is round-to-nearest-even)."""
    t = torch.from_numpy(a)
    return t.to(torch.bfloat16) if dtype == BF16 else t.clone()


def hidden_iid(seed: int, shape: LayerShape, T: int, tag="x") -> torch.Tensor:
    """T hidden states x ~ N(0, 1), [T, d] in the layer dtype."""
    return as_dtype(normal_f32(seed, (shape.name, tag), T * shape.d).reshape(T, shape.d), shape.dtype)


def ar1_streams(seed: int, shape: LayerShape, steps: int, rows: int, layer: int = 0,
                rho: float = 0.8) -> torch.Tensor:
    """Decode hidden states, [steps, rows, d]: one AR(1) stream per (layer, row)."""
    d = shape.d
    eps = normal_f32(seed, (shape.name, "ar1", layer), steps * rows * d).reshape(steps, rows, d)
    x = np.empty_like(eps)
    x[0] = eps[0] / np.float32(math.sqrt(1.0 - rho * rho))
    r = np.float32(rho)
    for t in range(1, steps):
        np.multiply(x[t - 1], r, out=x[t])
        x[t] += eps[t]
    return as_dtype(x, shape.dtype)


def router_weight(seed: int, shape: LayerShape, layer: int = 0) -> torch.Tensor:
    """Router weight W [E, d] ~ N(0, 0.02^2)."""
    a = normal_f32(seed, (shape.name, "router", layer), shape.E * shape.d, 0.02)
    return as_dtype(a.reshape(shape.E, shape.d), shape.dtype)


def norm_weight(seed: int, shape: LayerShape, layer: int = 0) -> torch.Tensor:
    """RMSNorm scale gamma [d] ~ 1 + N(0, 0.1^2) in the layer dtype."""
    a = normal_f32(seed, (shape.name, "norm", layer), shape.d, 0.1) + np.float32(1.0)
    return as_dtype(a, shape.dtype)


def residual_stream(seed: int, shape: LayerShape, steps: int, rows: int) -> torch.Tensor:
    """Stream entering the first block of a chained stack, [steps, rows, d] fp32: the AR(1)
    decode recipe (rounded to the layer dtype, as token embeddings are stored), widened to fp32."""
    return ar1_streams(seed, shape, steps, rows, layer=-1).float()


def expert_block(seed: int, shape: LayerShape, expert, layer: int = 0) -> torch.Tensor:
    """One packed expert [W1 (w x d) | W3 (w x d) | W2 (d x w)] as a flat tensor, N(0, 0.02^2).

    ``expert`` is an int for routed experts or ("shared", s) for shared experts.
    """
    a = normal_f32(seed, (shape.name, "expert", layer, expert), shape.expert_elems, 0.02)
    return as_dtype(a, shape.dtype)


def lora_block(seed: int, shape: LayerShape, expert, rank: int = 8, layer: int = 0,
               std_a: float = 0.02, std_b: float = 0.05) -> torch.Tensor:
    """Packed LoRA adapter of one expert, [A1 (r x d) | B1 (w x r) | A3 (r x d) | B3 (w x r) |
    A2 (r x w) | B2 (d x r)]; A ~ N(0, std_a^2), B ~ N(0, std_b^2) (trained adapters: B != 0)."""
    d, w, r = shape.d, shape.w, rank
    sizes = [r * d, w * r, r * d, w * r, r * w, d * r]
    parts = []
    for i, n in enumerate(sizes):
        parts.append(normal_f32(seed, (shape.name, "lora", layer, expert, rank, i), n,
                                std_a if i % 2 == 0 else std_b))
    return as_dtype(np.concatenate(parts), shape.dtype)


def split_lora(block: torch.Tensor, shape: LayerShape, rank: int = 8):
    """View a packed LoRA block as (A1, B1, A3, B3, A2, B2)."""
    d, w, r = shape.d, shape.w, rank
    shapes = [(r, d), (w, r), (r, d), (w, r), (r, w), (d, r)]
    out, o = [], 0
    for rr, cc in shapes:
        out.append(block[o:o + rr * cc].view(rr, cc))
        o += rr * cc
    return tuple(out)


def split_expert(block: torch.Tensor, shape: LayerShape):
    """View a packed expert block as (W1 [w,d], W3 [w,d], W2 [d,w])."""
    w, d = shape.w, shape.d
    b = block.reshape(-1)
    return (b[: w * d].view(w, d), b[w * d: 2 * w * d].view(w, d), b[2 * w * d:].view(d, w))


def keep_mask(seed: int, E: int, keep: int, layer: int = 0, tag="mask") -> np.ndarray:
    """Binary mask with exactly ``keep`` ones: the first ``keep`` ids of a seeded Fisher-Yates shuffle."""
    g = np.random.Generator(np.random.Philox(key=_key(seed, tag, E, keep, layer)))
    ids = np.arange(E)
    for i in range(E - 1, 0, -1):
        j = int(g.integers(0, i + 1))
        ids[i], ids[j] = ids[j], ids[i]
    m = np.zeros(E, np.uint8)
    m[ids[:keep]] = 1
    return m


def prior_from_mask(mask: np.ndarray, gamma: float = 2.0) -> np.ndarray:
    """Stand-in learned prior: pi = softmax(gamma * m), fp32, every entry > 0."""
    a = gamma * np.asarray(mask, np.float64)
    e = np.exp(a - a.max())
    return (e / e.sum()).astype(np.float32)


def uniforms(seed: int, shape, tag="u") -> np.ndarray:
    """fp32 uniforms strictly inside (0, 1) (for the mask sampler's Gumbel keys)."""
    g = np.random.Generator(np.random.Philox(key=_key(seed, tag, tuple(np.atleast_1d(shape)))))
    u = g.random(size=shape, dtype=np.float64)
    return np.clip(u, 2.0 ** -24, 1 - 2.0 ** -24).astype(np.float32)


def mask_from_ids(E: int, ids) -> np.ndarray:
    m = np.zeros(E, np.uint8)
    m[list(ids)] = 1
    return m


@dataclass
class LayerWeights:
    """Weights of one MoE layer, as CPU tensors in the layer dtype."""
    shape: LayerShape
    router: torch.Tensor
    experts: list = field(default_factory=list)   # E packed blocks
    shared: list = field(default_factory=list)    # S packed blocks


def layer_weights(seed: int, shape: LayerShape, layer: int = 0, experts=None,
                  pin: bool = False) -> LayerWeights:
    """Router + the listed routed experts (default all) + all shared experts of one layer."""
    ids = range(shape.E) if experts is None else experts
    lw = LayerWeights(shape, router_weight(seed, shape, layer))
    for e in range(shape.E):
        if e in ids:
            b = expert_block(seed, shape, e, layer)
            lw.experts.append(b.pin_memory() if pin else b)
        else:
            lw.experts.append(None)
    for s in range(shape.n_shared):
        b = expert_block(seed, shape, ("shared", s), layer)
        lw.shared.append(b.pin_memory() if pin else b)
    return lw


def random_ids(seed: int, steps: int, T: int, K: int, E: int, hot=None, p_hot=0.8, tag="ids"):
    """Synthetic routing decisions for cache tests: [steps, T, K] int32, K distinct ids per token.

    With ``hot`` given, each pick comes from the hot set with probability ``p_hot``.
    """
    g = np.random.Generator(np.random.Philox(key=_key(seed, tag, steps, T, K, E)))
    out = np.empty((steps, T, K), np.int32)
    hot = None if hot is None else np.asarray(sorted(hot))
    for s in range(steps):
        for t in range(T):
            chosen = []
            while len(chosen) < K:
                if hot is not None and g.random() < p_hot:
                    e = int(hot[g.integers(0, len(hot))])
                else:
                    e = int(g.integers(0, E))
                if e not in chosen:
                    chosen.append(e)
            out[s, t] = chosen
    return out
