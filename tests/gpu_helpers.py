"""Shared helpers of the GPU parity tests: inputs on the device, oracle views, comparisons.

Tolerances (written here, used by every parity test):
* expert ids: bit-exact, except tokens whose K-th and (K+1)-th oracle scores are within a relative
  1e-4 of each other (near ties, counted); there the chosen set must still consist of experts whose
  score is within that band of the K-th, and the order may differ where adjacent selected scores are
  within the band;
* gates (fp32): |g - g_ref| <= 1e-5 + 1e-4 |g_ref|, for the set the GPU chose;
* layer outputs: row-wise max_j |y - y_ref| / max_j |y_ref| <= 2e-2 in bf16, <= 1e-4 in fp32.
"""
from __future__ import annotations

import functools

import numpy as np
import torch

import oracle
from paper_2609_34077_gb300 import inputs as I

NEAR_TIE = 1e-4
TOL_BF16 = 2e-2
TOL_F32 = 1e-4


def f64(t: torch.Tensor) -> np.ndarray:
    return t.detach().cpu().double().numpy()


@functools.lru_cache(maxsize=8)
def weights(shape: I.LayerShape, seed: int = 0, layer: int = 0):
    return I.layer_weights(seed, shape, layer)


def expert_triples(lw: I.LayerWeights, shape):
    return [None if b is None else tuple(f64(t) for t in I.split_expert(b, shape))
            for b in lw.experts]


def shared_triples(lw: I.LayerWeights, shape):
    return [tuple(f64(t) for t in I.split_expert(b, shape)) for b in lw.shared]


def check_routing(idx_gpu, gate_gpu, ref, gate_mode):
    """Compare GPU routing with the oracle's under the near-tie rule. Returns (n_flagged, n_swapped)."""
    idx = idx_gpu.cpu().numpy()
    gate = gate_gpu.cpu().double().numpy()
    T, K = idx.shape
    s, p = ref["s"], ref["p"]
    flagged = swapped = 0
    for t in range(T):
        exact = list(idx[t]) == list(ref["idx"][t])
        near_k = ref["gap_k"][t] < NEAR_TIE
        near_in = ref["gap_in"][t] < NEAR_TIE
        if near_k or near_in:
            flagged += 1
        if not exact:
            assert near_k or near_in, f"token {t}: {idx[t]} != {ref['idx'][t]} outside a near tie"
            assert len(set(idx[t])) == K
            sk = s[t, ref["idx"][t][K - 1]]
            for e in idx[t]:
                assert s[t, e] >= sk * (1 - NEAR_TIE), f"token {t}: expert {e} is not near the K-th"
            if set(idx[t]) != set(ref["idx"][t]):
                assert near_k
                swapped += 1
        # gates for the set the GPU chose, from the oracle's p
        pa = p[t, idx[t]]
        g_ref = pa / pa.sum() if gate_mode == I.GATE_RENORM else pa
        np.testing.assert_allclose(gate[t], g_ref, rtol=1e-4, atol=1e-5, err_msg=f"gates of token {t}")
    return flagged, swapped


def check_output(y_gpu, y_ref, tol, what=""):
    row, fro = oracle.ffn.rel_err_rows(f64(y_gpu), y_ref)
    assert row.max() <= tol, f"{what}: max row error {row.max():.3e} > {tol} (frobenius {fro:.3e})"
    return row.max(), fro


class _DevArray:
    """Wraps a raw device address for torch.as_tensor (CUDA array interface, the test only reads it)."""

    def __init__(self, ptr, n, typestr):
        self.__cuda_array_interface__ = dict(shape=(n,), typestr=typestr, data=(int(ptr), False),
                                             version=3, strides=None)


def device_view(ptr, n, dtype=torch.int32):
    """Tensor view of n elements at a device address returned by the library."""
    typestr = {torch.int32: "<i4", torch.uint8: "|u1", torch.float32: "<f4"}[dtype]
    return torch.as_tensor(_DevArray(ptr, n, typestr), device="cuda")
