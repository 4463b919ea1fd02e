"""Stage-1 mask machinery on the GPU against the oracle, through the C ABI (Section 3.2 Eq. stage1
and Eq. ste): mask sampling, gate gradients from a forward's expert outputs, the straight-through
mask gradient, and one full Stage-1 step chained through them."""
import numpy as np
import pytest
import torch

import oracle
from paper_2609_34077_gb300 import inputs as I
from paper_2609_34077_gb300 import mcft as M
from tests.gpu_helpers import NEAR_TIE, TOL_BF16, expert_triples, f64, weights

pytestmark = pytest.mark.gpu
DEV = "cuda"
SMALL = I.LayerShape("mask-small", d=256, E=16, K=4, w=128, n_shared=0, gate=I.GATE_RENORM,
                     dtype=I.BF16, cache_slots=6, keep=12)


@pytest.mark.parametrize("L,E,keep", [(32, 8, 6), (26, 64, 48), (32, 8, 4), (26, 64, 16), (3, 5, 1)])
def test_mask_sample_parity(L, E, keep):
    m_t = np.random.default_rng(L * E).standard_normal((L, E)).astype(np.float32)
    u = I.uniforms(L + E + keep, (L, E))
    mask, pi = M.mcft_mask_sample(torch.from_numpy(m_t).to(DEV), torch.from_numpy(u).to(DEV), keep)
    M.mcft_device_error()
    ref_mask, ref_pi, keys = oracle.mask.sample_mask(m_t, u, keep)
    np.testing.assert_allclose(pi.cpu().numpy(), ref_pi, rtol=1e-5)
    got = mask.cpu().numpy()
    assert np.all(got.sum(axis=1) == keep)
    for l in range(L):
        if not np.array_equal(got[l], ref_mask[l]):  # only when the E'-th keys nearly tie
            ks = np.sort(keys[l])[::-1]
            assert abs(ks[keep - 1] - ks[keep]) < 1e-5 * max(1.0, abs(ks[keep - 1]))


def _forward(shape, T, seed):
    lw = weights(shape, seed)
    x = I.hidden_iid(seed, shape, T)
    ids = I.random_ids(seed, 1, T, shape.K, shape.E, hot=range(shape.keep))[0]
    gate = np.random.default_rng(seed).uniform(0.05, 1.0, (T, shape.K)).astype(np.float32)
    desc = M.desc_of(shape)
    ws = torch.empty(M.mcft_moe_workspace_size(desc, T), dtype=torch.uint8, device=DEV)
    M.mcft_moe_forward(desc, x.to(DEV), torch.from_numpy(ids).to(DEV), torch.from_numpy(gate).to(DEV),
                       [b.to(DEV) for b in lw.experts], workspace=ws)
    return lw, x, ids, gate, desc, ws


@pytest.mark.parametrize("T", [1, 16, 64, 300])  # decode GEMV and tcgen05 paths
def test_gate_grad_parity(T):
    sh = SMALL
    lw, x, ids, gate, desc, ws = _forward(sh, T, 80 + T)
    dy = I.hidden_iid(81 + T, sh, T, tag="dy")
    dg = M.mcft_gate_grad(desc, dy.to(DEV), ws)
    M.mcft_device_error()
    ex = expert_triples(lw, sh)
    outs = np.stack([np.stack([oracle.ffn.expert(f64(x)[t:t + 1], *ex[ids[t, k]])[0]
                               for k in range(sh.K)]) for t in range(T)])
    ref = oracle.mask.gate_grad(f64(dy), outs)
    err = np.abs(dg.cpu().double().numpy() - ref).max() / np.abs(ref).max()
    assert err <= TOL_BF16, err


@pytest.mark.parametrize("gate_mode", [I.GATE_RENORM, I.GATE_PLAIN])
@pytest.mark.parametrize("T,E,K", [(1, 8, 2), (512, 8, 2), (4096, 8, 2), (300, 64, 6)])
def test_mask_grad_parity(gate_mode, T, E, K):
    g = np.random.default_rng(T + E + K + gate_mode)
    ids = I.random_ids(T + E, 1, T, K, E)[0]
    gate = g.uniform(0.05, 1.0, (T, K)).astype(np.float32)
    dgate = g.standard_normal((T, K)).astype(np.float32)
    pi = oracle.mask.softmax(g.standard_normal(E)).astype(np.float32)
    desc = M.LayerDesc(256, E, K, 128, 0, gate_mode, M.MCFT_BF16)
    args = [torch.from_numpy(a).to(DEV) for a in (ids, gate, dgate, pi)]
    dm, dmt = M.mcft_mask_grad(desc, *args)
    dm2, dmt2 = M.mcft_mask_grad(desc, *args, dm_tilde=dmt.clone(), accumulate=True)
    M.mcft_device_error()
    ref_dm = oracle.mask.mask_grad(ids, gate, dgate, gate_mode, E)
    ref_dmt = oracle.mask.mask_tilde_grad(pi, ref_dm)
    scale = max(np.abs(ref_dm).max(), 1e-30)
    np.testing.assert_allclose(dm.cpu().double().numpy(), ref_dm, atol=1e-5 * scale, rtol=1e-4)
    np.testing.assert_allclose(dmt.cpu().double().numpy(), ref_dmt, atol=1e-5 * scale, rtol=1e-4)
    np.testing.assert_allclose(dmt2.cpu().double().numpy(), 2 * ref_dmt, atol=2e-5 * scale, rtol=1e-4)
    assert abs(dmt.sum().item()) <= 1e-4 * scale  # rows of the softmax Jacobian sum to zero


def test_stage1_step_end_to_end():
    """Sample the mask from m~, route with the hard mask, run the layer, take dL/dy = y (the loss
    0.5 |y|^2), and carry the gradient to m~: GPU chain against the oracle chain."""
    sh, T = SMALL, 96
    lw = weights(sh, 90)
    x = I.hidden_iid(90, sh, T)
    m_t = np.random.default_rng(90).standard_normal((1, sh.E)).astype(np.float32)
    u = I.uniforms(90, (1, sh.E))
    desc = M.desc_of(sh)
    mask, pi = M.mcft_mask_sample(torch.from_numpy(m_t).to(DEV), torch.from_numpy(u).to(DEV), sh.keep)
    ref_mask, ref_pi, _ = oracle.mask.sample_mask(m_t, u, sh.keep)
    assert np.array_equal(mask.cpu().numpy(), ref_mask)
    idx, gate = M.mcft_route(desc, x.to(DEV), lw.router.to(DEV), M.MCFT_ROUTE_HARD_MASK,
                             mask=ref_mask[0])
    ws = torch.empty(M.mcft_moe_workspace_size(desc, T), dtype=torch.uint8, device=DEV)
    y = M.mcft_moe_forward(desc, x.to(DEV), idx, gate, [b.to(DEV) for b in lw.experts], workspace=ws)
    dg = M.mcft_gate_grad(desc, y, ws)
    dm, dmt = M.mcft_mask_grad(desc, idx, gate, dg, pi[0])
    M.mcft_device_error()
    # oracle chain on its own routing
    r = oracle.routing.route(f64(x), f64(lw.router), sh.K, M.MCFT_ROUTE_HARD_MASK, sh.gate,
                             mask=ref_mask[0])
    assert np.array_equal(idx.cpu().numpy(), r["idx"]) or np.any(r["gap_k"] < NEAR_TIE)
    ex = expert_triples(lw, sh)
    y_ref = oracle.ffn.moe_layer(f64(x), r["idx"], r["gate"], ex)
    outs = np.stack([np.stack([oracle.ffn.expert(f64(x)[t:t + 1], *ex[r["idx"][t, k]])[0]
                               for k in range(sh.K)]) for t in range(T)])
    dg_ref = oracle.mask.gate_grad(y_ref, outs)
    dm_ref = oracle.mask.mask_grad(r["idx"], r["gate"], dg_ref, sh.gate, sh.E)
    dmt_ref = oracle.mask.mask_tilde_grad(ref_pi[0], dm_ref)
    # masked experts never get a gradient through the gates (they are never active)
    assert np.all(dm.cpu().numpy()[ref_mask[0] == 0] == 0)
    scale = np.abs(dmt_ref).max()
    assert np.abs(dmt.cpu().double().numpy() - dmt_ref).max() <= 3e-2 * scale


def test_gate_grad_mixtral_full_size():
    """Gate gradients of a Mixtral-shaped fine-tuning batch of 4096 tokens (tcgen05 forward, the
    size the bench times): every token against the oracle's <dL/dy_t, F_e(x_t)>, with each
    expert's outputs from the oracle's expert on the rows routed to it."""
    sh, T = I.MIXTRAL, 4096
    lw = weights(sh)
    x = I.hidden_iid(83, sh, T)
    ids = I.random_ids(83, 1, T, sh.K, sh.E, hot=range(6), p_hot=1.0)[0]
    gate = np.random.default_rng(83).uniform(0.05, 1.0, (T, sh.K)).astype(np.float32)
    desc = M.desc_of(sh)
    ws = torch.empty(M.mcft_moe_workspace_size(desc, T), dtype=torch.uint8, device=DEV)
    M.mcft_moe_forward(desc, x.to(DEV), torch.from_numpy(ids).to(DEV),
                       torch.from_numpy(gate).to(DEV),
                       [b.to(DEV) if e < 6 else None for e, b in enumerate(lw.experts)], workspace=ws)
    dy = I.hidden_iid(84, sh, T, tag="dy")
    dg = M.mcft_gate_grad(desc, dy.to(DEV), ws).cpu().double().numpy()
    M.mcft_device_error()
    ex = [tuple(f64(t) for t in I.split_expert(lw.experts[e], sh)) if e < 6 else None
          for e in range(sh.E)]
    xs = f64(x)
    outs = np.zeros((T, sh.K, sh.d))
    for k in range(sh.K):
        for e in np.unique(ids[:, k]):
            r = np.nonzero(ids[:, k] == e)[0]
            outs[r, k] = oracle.ffn.expert(xs[r], *ex[int(e)])
    ref = oracle.mask.gate_grad(f64(dy), outs)
    err = np.abs(dg - ref).max() / np.abs(ref).max()
    assert err <= TOL_BF16, err
