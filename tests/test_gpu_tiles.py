"""The CTA-pair tile shape of the tensor-core expert GEMMs (mcft_set_tc_tiles): 256-row tiles whose
MMAs run over the shared memory of a 2-CTA cluster, with segments padded to 256 rows. The same
products are summed in the same order as on the one-CTA tiles, so the forward (Section 3.1, the
gated sum of SwiGLU experts) must give the same bits; the one-CTA path is itself compared with the
oracle on every row in test_gpu_layer.py, and one pair-tile forward is compared here too."""
import numpy as np
import pytest
import torch

from paper_2609_34077_gb300 import inputs as I
from paper_2609_34077_gb300 import mcft as M

pytestmark = pytest.mark.gpu
DEV = "cuda"


def _forward(desc, x, idx, gate, experts, shared, mode):
    """y and the per-kernel profile of one forward with tile mode `mode` (workspace sized under
    it); restores the default mode."""
    M.mcft_set_tc_tiles(mode)
    try:
        T = x.shape[0]
        ws = torch.empty(M.mcft_moe_workspace_size(desc, T), dtype=torch.uint8, device=DEV)
        M.mcft_profile_reset()
        M.mcft_profile_enable(True)
        y = M.mcft_moe_forward(desc, x, idx, gate, experts, shared, workspace=ws)
        M.mcft_profile_enable(False)
        prof = M.mcft_profile_read()
        M.mcft_device_error()
        return y, prof, ws.numel()
    finally:
        M.mcft_profile_enable(False)
        M.mcft_set_tc_tiles(M.MCFT_TC_TILES_ONE_CTA)


def _case(shape, T, seed, keep=None, hot=None, p_hot=None):
    """Routing from the router with a hard mask (keep experts) or seeded ids skewed to a few hot
    experts (ragged segments of very different sizes)."""
    kept = list(range(shape.E)) if keep is None else \
        [int(e) for e in np.nonzero(I.keep_mask(seed, shape.E, keep))[0]]
    lw = I.layer_weights(seed, shape, experts=kept)
    desc = M.desc_of(shape)
    x = I.hidden_iid(seed, shape, T).to(DEV)
    if keep is not None:
        mask = I.keep_mask(seed, shape.E, keep)
        idx, gate = M.mcft_route(desc, x, lw.router.to(DEV), M.MCFT_ROUTE_HARD_MASK, mask=mask)
    else:
        ids = I.random_ids(seed, 1, T, shape.K, shape.E, hot=hot, p_hot=p_hot)[0]
        g = np.random.default_rng(seed).uniform(0.05, 1.0, (T, shape.K)).astype(np.float32)
        idx, gate = torch.from_numpy(ids).to(DEV), torch.from_numpy(g).to(DEV)
    experts = [None if b is None else b.to(DEV) for b in lw.experts]
    shared = [b.to(DEV) for b in lw.shared]
    return desc, x, idx, gate, experts, shared


@pytest.mark.parametrize("shape,T,kw", [
    (I.MIXTRAL, 4096, dict(keep=4)),
    (I.MIXTRAL, 2100, dict(hot=[1, 6], p_hot=0.7)),
    (I.DSV2_LITE, 8192, dict(keep=48)),
], ids=["mixtral-T4096-keep4", "mixtral-T2100-skewed", "deepseek-T8192-keep48"])
def test_cta_pair_tiles_equal_one_cta_tiles_bitwise(shape, T, kw):
    desc, x, idx, gate, experts, shared = _case(shape, T, 120 + T, **kw)
    y1, p1, ws1 = _forward(desc, x, idx, gate, experts, shared, M.MCFT_TC_TILES_ONE_CTA)
    y2, p2, ws2 = _forward(desc, x, idx, gate, experts, shared, M.MCFT_TC_TILES_CTA_PAIR)
    # the pair layout (segments padded to 256 rows) and the pair kernels were used
    assert ws2 > ws1
    assert p2["gemm13_tc_pair"][0] == 1 and p2["gemm2_tc_pair"][0] == 1
    assert p2["gemm13_tc"][0] == 0 and p1["gemm13_tc_pair"][0] == 0
    assert torch.isfinite(y2).all()
    assert torch.equal(y1, y2), f"{shape.name} T={T}"


def test_cta_pair_tiles_against_the_oracle_every_row():
    """Mixtral-shaped T = 4096 (keep 4 of 8) on pair tiles, every row against the oracle."""
    from tests.test_gpu_layer import _prefill_full

    M.mcft_set_tc_tiles(M.MCFT_TC_TILES_CTA_PAIR)
    try:
        _prefill_full(I.MIXTRAL, 4, seed=93)
    finally:
        M.mcft_set_tc_tiles(M.MCFT_TC_TILES_ONE_CTA)


def test_small_layers_keep_one_cta_tiles():
    """Routed experts averaging fewer than 512 rows keep the one-CTA tiles under the pair mode."""
    desc, x, idx, gate, experts, shared = _case(I.MIXTRAL, 1024, 131, keep=4)
    y1, _, ws1 = _forward(desc, x, idx, gate, experts, shared, M.MCFT_TC_TILES_ONE_CTA)
    y2, p2, ws2 = _forward(desc, x, idx, gate, experts, shared, M.MCFT_TC_TILES_CTA_PAIR)
    assert ws2 == ws1 and p2["gemm13_tc_pair"][0] == 0 and p2["gemm13_tc"][0] == 1
    assert torch.equal(y1, y2)


def test_workspace_sized_for_one_cta_tiles_is_rejected_under_pairs():
    desc, x, idx, gate, experts, shared = _case(I.MIXTRAL, 4096, 132, keep=4)
    ws = torch.empty(M.mcft_moe_workspace_size(desc, 4096), dtype=torch.uint8, device=DEV)
    M.mcft_set_tc_tiles(M.MCFT_TC_TILES_CTA_PAIR)
    try:
        with pytest.raises(M.MCFTError):
            M.mcft_moe_forward(desc, x, idx, gate, experts, shared, workspace=ws)
    finally:
        M.mcft_set_tc_tiles(M.MCFT_TC_TILES_ONE_CTA)
    M.mcft_device_error()
