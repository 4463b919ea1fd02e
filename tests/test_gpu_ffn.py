"""GPU expert FFN + combine (permutation, SwiGLU experts, gated sum, shared experts) against the
oracle, through the C ABI. Section 3.1 Eq. topk. Routing is an input here (seeded ids and gates), so
these tests isolate the FFN path; the end-to-end layer tests chain routing in."""
import numpy as np
import pytest
import torch

import oracle
from paper_2609_34077_gb300 import inputs as I
from paper_2609_34077_gb300 import mcft as M
from tests.gpu_helpers import TOL_BF16, TOL_F32, check_output, expert_triples, f64, shared_triples, weights

pytestmark = pytest.mark.gpu
DEV = "cuda"

# small shapes that run every path with several tiles and ragged tails
SMALL_BF16 = I.LayerShape("small-bf16", d=512, E=8, K=2, w=384, n_shared=0, gate=I.GATE_RENORM,
                          dtype=I.BF16, cache_slots=4, keep=4)
SMALL_DS = I.LayerShape("small-ds", d=256, E=64, K=6, w=128, n_shared=2, gate=I.GATE_PLAIN,
                        dtype=I.BF16, cache_slots=12, keep=16)
SMALL_F32_SH = I.LayerShape("small-f32-shared", d=128, E=16, K=4, w=192, n_shared=2,
                            gate=I.GATE_PLAIN, dtype=I.F32, cache_slots=6, keep=8)


def _routing(shape, T, seed, hot=None):
    ids = I.random_ids(seed, 1, T, shape.K, shape.E, hot=hot, p_hot=0.8)[0]
    g = np.random.default_rng(seed).uniform(0.05, 1.0, (T, shape.K)).astype(np.float32)
    return torch.from_numpy(ids), torch.from_numpy(g)


def _forward(shape, x, idx, gate, lw, experts_dev=None):
    desc = M.desc_of(shape)
    ex = experts_dev if experts_dev is not None else [b.to(DEV) for b in lw.experts]
    sh = [b.to(DEV) for b in lw.shared]
    y = M.mcft_moe_forward(desc, x.to(DEV), idx.to(DEV), gate.to(DEV), ex, sh)
    M.mcft_device_error()
    return y


def _reference(shape, x, idx, gate, lw, rows=None):
    rows = np.arange(x.shape[0]) if rows is None else rows
    return oracle.ffn.moe_layer(f64(x)[rows], idx.numpy()[rows], gate.double().numpy()[rows],
                                expert_triples(lw, shape), shared_triples(lw, shape))


@pytest.mark.parametrize("T", [1, 7, 64, 130])
def test_ffn_tiny_fp32(T):
    sh = I.TINY
    lw = weights(sh)
    x = I.hidden_iid(5, sh, T)
    idx, gate = _routing(sh, T, 5)
    y = _forward(sh, x, idx, gate, lw)
    check_output(y, _reference(sh, x, idx, gate, lw), TOL_F32, "tiny fp32")


@pytest.mark.parametrize("T", [1, 33, 200])
def test_ffn_fp32_shared_experts(T):
    sh = SMALL_F32_SH
    lw = weights(sh)
    x = I.hidden_iid(6, sh, T)
    idx, gate = _routing(sh, T, 6)
    y = _forward(sh, x, idx, gate, lw)
    check_output(y, _reference(sh, x, idx, gate, lw), TOL_F32, "fp32 + shared")


@pytest.mark.parametrize("shape", [SMALL_BF16, SMALL_DS], ids=lambda s: s.name)
@pytest.mark.parametrize("T", [1, 5, 16, 64, 65, 300, 1000])
def test_ffn_bf16_paths(shape, T):
    """T <= 64: HBM-streaming GEMV path; T > 64: tcgen05 grouped GEMM path (tiles of 128 rows,
    ragged tails, experts with no tokens)."""
    lw = weights(shape)
    x = I.hidden_iid(7, shape, T)
    idx, gate = _routing(shape, T, 7, hot=range(shape.keep))
    y = _forward(shape, x, idx, gate, lw)
    check_output(y, _reference(shape, x, idx, gate, lw), TOL_BF16, f"{shape.name} T={T}")


def test_ffn_tc_single_expert_all_tokens():
    sh = SMALL_BF16
    lw = weights(sh)
    T = 517
    x = I.hidden_iid(8, sh, T)
    idx = torch.tensor([[3, 5]] * T, dtype=torch.int32)
    gate = torch.full((T, 2), 0.5)
    experts = [None] * sh.E
    experts[3], experts[5] = lw.experts[3].to(DEV), lw.experts[5].to(DEV)
    y = _forward(sh, x, idx, gate, lw, experts_dev=experts)
    check_output(y, _reference(sh, x, idx, gate, lw), TOL_BF16, "one pair of experts")


@pytest.mark.parametrize("batch", [1, 16])
def test_ffn_mixtral_decode_full_size(batch):
    sh = I.MIXTRAL
    lw = weights(sh)
    x = I.ar1_streams(9, sh, 1, batch)[0]
    idx, gate = _routing(sh, batch, 9, hot=range(4))
    y = _forward(sh, x, idx, gate, lw)
    check_output(y, _reference(sh, x, idx, gate, lw), TOL_BF16, f"mixtral decode b={batch}")


@pytest.mark.parametrize("batch", [1, 8, 64])
def test_ffn_deepseek_decode_full_size(batch):
    sh = I.DSV2_LITE
    lw = weights(sh)
    x = I.ar1_streams(10, sh, 1, batch)[0]
    idx, gate = _routing(sh, batch, 10, hot=range(16))
    y = _forward(sh, x, idx, gate, lw)
    check_output(y, _reference(sh, x, idx, gate, lw), TOL_BF16, f"deepseek decode b={batch}")


def test_ffn_mixtral_prefill_full_size():
    """T = 4096 tokens, hard mask keeping 4 of 8 experts, seeded ids folded onto the kept set
    (unbalanced loads): every output row matches the oracle."""
    sh = I.MIXTRAL
    lw = weights(sh)
    T = 4096
    x = I.hidden_iid(11, sh, T)
    kept = np.nonzero(I.keep_mask(11, sh.E, 4))[0]
    idx, gate = _routing(sh, T, 11, hot=kept)
    idx = torch.from_numpy(np.where(np.isin(idx.numpy(), kept), idx.numpy(), kept[0]).astype(np.int32))
    # keep K distinct ids per token after the projection onto the kept set
    for t in range(T):
        if idx[t, 0] == idx[t, 1]:
            idx[t, 1] = int(kept[(list(kept).index(int(idx[t, 0])) + 1) % len(kept)])
    y = _forward(sh, x, idx, gate, lw)
    assert torch.isfinite(y.float()).all()
    check_output(y, _reference(sh, x, idx, gate, lw), TOL_BF16, "mixtral prefill, every row")


def test_ffn_empty_and_bad_ids():
    sh = SMALL_BF16
    lw = weights(sh)
    desc = M.desc_of(sh)
    ex = [b.to(DEV) for b in lw.experts]
    x = I.hidden_iid(12, sh, 3000).to(DEV)
    y0 = torch.empty((0, sh.d), dtype=torch.bfloat16, device=DEV)
    M.mcft_moe_forward(desc, x[:0], torch.empty((0, 2), dtype=torch.int32, device=DEV),
                       torch.empty((0, 2), device=DEV), ex, y=y0)
    M.mcft_device_error()
    # an id out of range: the device error word is set and y is left untouched (every decode
    # kernel variant: 1, 16 and 64 tokens; the tensor-core path; and 6000 assignments, which the
    # chunked permutation handles)
    for T in (1, 16, 64, 100, 3000):
        idx = torch.zeros((T, 2), dtype=torch.int32, device=DEV)
        idx[:, 1] = 1
        idx[T // 2, 1] = sh.E
        y = torch.full((T, sh.d), 7.0, dtype=torch.bfloat16, device=DEV)
        M.mcft_moe_forward(desc, x[:T], idx, torch.ones((T, 2), device=DEV), ex, y=y)
        with pytest.raises(M.MCFTError) as ei:
            M.mcft_device_error()
        assert ei.value.status == M.MCFT_ERR_INVALID
        assert torch.all(y == 7.0)
    # a selected expert with no weights
    for T in (1, 16, 64, 100, 3000):
        idx = torch.zeros((T, 2), dtype=torch.int32, device=DEV)
        idx[:, 1] = 2
        missing = list(ex)
        missing[2] = None
        y = torch.full((T, sh.d), 7.0, dtype=torch.bfloat16, device=DEV)
        M.mcft_moe_forward(desc, x[:T], idx, torch.ones((T, 2), device=DEV), missing, y=y)
        with pytest.raises(M.MCFTError):
            M.mcft_device_error()
        assert torch.all(y == 7.0)
    M.mcft_device_error()


@pytest.mark.parametrize("shape,T", [(SMALL_BF16, 2049), (SMALL_BF16, 2500), (SMALL_DS, 700)],
                         ids=["mix-4098", "mix-5000", "ds-4200"])
def test_ffn_chunked_permutation(shape, T):
    """Just above 4096 assignments the permutation runs in chunks (ragged: 820 to 1000
    assignments each, shared-expert rows filled by every chunk's CTA); every output row matches
    the oracle."""
    lw = weights(shape)
    x = I.hidden_iid(13, shape, T)
    idx, gate = _routing(shape, T, 13, hot=range(shape.keep))
    y = _forward(shape, x, idx, gate, lw)
    check_output(y, _reference(shape, x, idx, gate, lw), TOL_BF16, f"{shape.name} T={T}")
