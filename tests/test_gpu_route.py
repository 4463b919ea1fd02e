"""GPU routing (router GEMV + mask / prior + Top-K + gates) against the oracle, through the C ABI.

Section 3.1 Eq. topk, Section 3.2 Eq. stage1 (hard mask) and Eq. inference (soft prior)."""
import numpy as np
import pytest
import torch

import oracle
from paper_2609_34077_gb300 import inputs as I
from paper_2609_34077_gb300 import mcft as M
from tests.gpu_helpers import check_routing, f64, weights

pytestmark = pytest.mark.gpu
DEV = "cuda"
MODES = {"topk": M.MCFT_ROUTE_TOPK, "hard": M.MCFT_ROUTE_HARD_MASK, "soft": M.MCFT_ROUTE_SOFT_PRIOR}


def _mode_args(shape, mode, seed=0):
    mask = I.keep_mask(seed, shape.E, shape.keep) if shape is not I.TINY else I.mask_from_ids(8, range(4))
    if mode == M.MCFT_ROUTE_HARD_MASK:
        return dict(mask=mask)
    if mode == M.MCFT_ROUTE_SOFT_PRIOR:
        return dict(prior=I.prior_from_mask(mask))
    return {}


def _run(shape, x, mode, **kw):
    lw = weights(shape)
    desc = M.desc_of(shape)
    idx, gate = M.mcft_route(desc, x.to(DEV), lw.router.to(DEV), mode, **kw)
    M.mcft_device_error()
    ref = oracle.routing.route(f64(x), f64(lw.router), shape.K, mode, shape.gate,
                               mask=kw.get("mask"), prior=kw.get("prior"))
    return idx, gate, ref


@pytest.mark.parametrize("shape", [I.TINY, I.MIXTRAL, I.DSV2_LITE], ids=lambda s: s.name)
@pytest.mark.parametrize("mode", list(MODES.values()), ids=list(MODES))
@pytest.mark.parametrize("T", [1, 16, 64, 65, 333])
def test_route_parity(shape, mode, T):
    x = I.hidden_iid(1, shape, T)
    kw = _mode_args(shape, mode)
    idx, gate, ref = _run(shape, x, mode, **kw)
    check_routing(idx, gate, ref, shape.gate)
    if mode == M.MCFT_ROUTE_HARD_MASK:
        assert np.all(kw["mask"][idx.cpu().numpy()] == 1)


def test_route_prefill_full_size_hard_mask():
    """Mixtral-shaped masked fine-tuning forward: T = 8 x 512 = 4096 tokens, keep 4 of 8."""
    sh = I.MIXTRAL
    x = I.hidden_iid(2, sh, 4096)
    kw = _mode_args(sh, M.MCFT_ROUTE_HARD_MASK, seed=2)
    idx, gate, ref = _run(sh, x, M.MCFT_ROUTE_HARD_MASK, **kw)
    flagged, swapped = check_routing(idx, gate, ref, sh.gate)
    assert flagged < 4096 // 100
    assert np.all(kw["mask"][idx.cpu().numpy()] == 1)


def test_route_prefill_full_size_dsv2_soft_prior():
    """DeepSeek-V2-Lite-shaped T = 4096 (the tensor-core tiles: 8 column tiles of 8 experts, one
    warp each, over the whole contraction), soft prior of a keep-16-of-64 mask, plus a ragged
    tail of 4096 + 7 tokens in top-k mode."""
    sh = I.DSV2_LITE
    for T, mode in ((4096, M.MCFT_ROUTE_SOFT_PRIOR), (4103, M.MCFT_ROUTE_TOPK)):
        x = I.hidden_iid(5, sh, T)
        kw = _mode_args(sh, mode, seed=5)
        idx, gate, ref = _run(sh, x, mode, **kw)
        flagged, swapped = check_routing(idx, gate, ref, sh.gate)
        assert flagged < T // 100


@pytest.mark.parametrize("shape,batch", [(I.MIXTRAL, 16), (I.DSV2_LITE, 64)], ids=["mixtral-b16", "dsv2-b64"])
def test_route_decode_stream_full_size(shape, batch):
    """512 decode steps of AR(1) hidden states (rho = 0.8) routed with the soft prior."""
    x = I.ar1_streams(3, shape, 512, batch).reshape(512 * batch, shape.d)
    kw = _mode_args(shape, M.MCFT_ROUTE_SOFT_PRIOR, seed=3)
    idx, gate, ref = _run(shape, x, M.MCFT_ROUTE_SOFT_PRIOR, **kw)
    flagged, swapped = check_routing(idx, gate, ref, shape.gate)
    assert flagged <= x.shape[0] // 100


def test_route_uniform_prior_equals_plain_topk():
    sh = I.DSV2_LITE
    x = I.hidden_iid(4, sh, 256)
    a, ga, _ = _run(sh, x, M.MCFT_ROUTE_TOPK)
    b, gb, _ = _run(sh, x, M.MCFT_ROUTE_SOFT_PRIOR, prior=np.full(64, 1 / 64, np.float32))
    assert torch.equal(a, b) and torch.equal(ga, gb)


def test_route_empty_and_exact_ties():
    sh = I.TINY
    desc = M.desc_of(sh)
    lw = weights(sh)
    x = torch.zeros((3, sh.d), dtype=torch.float32, device=DEV)
    idx, gate = M.mcft_route(desc, x, lw.router.to(DEV), M.MCFT_ROUTE_TOPK)
    assert idx.cpu().tolist() == [[0, 1]] * 3
    assert torch.allclose(gate.cpu(), torch.full((3, 2), 0.5))
    idx, gate = M.mcft_route(desc, x[:0], lw.router.to(DEV), M.MCFT_ROUTE_TOPK)
    assert idx.shape == (0, 2)
    M.mcft_device_error()
