"""Stage-2 forward with LoRA adapters on the experts (Section 3.2; rank 8 / alpha 16, Appendix B)
against the oracle, through the C ABI, on the three FFN paths: fp32 (CUDA cores), bf16 decode
(T <= 64, HBM-streaming GEMV) and bf16 prefill (T > 64, tcgen05 grouped GEMM)."""
import numpy as np
import pytest
import torch

import oracle
from paper_2609_34077_gb300 import inputs as I
from paper_2609_34077_gb300 import mcft as M
from tests.gpu_helpers import TOL_BF16, TOL_F32, check_output, expert_triples, f64, shared_triples, weights

pytestmark = pytest.mark.gpu
DEV = "cuda"

TINY_SH = I.LayerShape("lora-f32-shared", d=128, E=8, K=2, w=192, n_shared=1, gate=I.GATE_RENORM,
                       dtype=I.F32, cache_slots=4, keep=4)
BF_MIX = I.LayerShape("lora-bf16-mix", d=512, E=8, K=2, w=384, n_shared=0, gate=I.GATE_RENORM,
                      dtype=I.BF16, cache_slots=4, keep=4)
BF_DS = I.LayerShape("lora-bf16-ds", d=256, E=16, K=4, w=256, n_shared=2, gate=I.GATE_PLAIN,
                     dtype=I.BF16, cache_slots=6, keep=8)


def _case(shape, T, rank, seed, with_adapter):
    lw = weights(shape, seed)
    x = I.hidden_iid(seed + 1, shape, T)
    ids = I.random_ids(seed + 2, 1, T, shape.K, shape.E, hot=range(shape.keep))[0]
    gate = np.random.default_rng(seed + 3).uniform(0.05, 1.0, (T, shape.K)).astype(np.float32)
    ad = [I.lora_block(seed, shape, e, rank) if with_adapter(e) else None for e in range(shape.E)]
    sad = [I.lora_block(seed, shape, ("shared", s), rank) for s in range(shape.n_shared)]
    desc = M.desc_of(shape)
    y = M.mcft_moe_forward_lora(
        desc, x.to(DEV), torch.from_numpy(ids).to(DEV), torch.from_numpy(gate).to(DEV),
        [b.to(DEV) for b in lw.experts], [b.to(DEV) for b in lw.shared],
        [None if b is None else b.to(DEV) for b in ad], [b.to(DEV) for b in sad], rank, 16.0 / rank)
    M.mcft_device_error()
    split = lambda b: None if b is None else tuple(f64(t) for t in I.split_lora(b, shape, rank))
    ref = oracle.ffn.moe_layer(f64(x), ids, gate.astype(np.float64), expert_triples(lw, shape),
                               shared_triples(lw, shape), lora=[split(b) for b in ad],
                               shared_lora=[split(b) for b in sad], lora_scale=16.0 / rank)
    base = oracle.ffn.moe_layer(f64(x), ids, gate.astype(np.float64), expert_triples(lw, shape),
                                shared_triples(lw, shape))
    return y, ref, base


@pytest.mark.parametrize("shape,T", [(TINY_SH, 7), (TINY_SH, 100), (BF_MIX, 1), (BF_MIX, 16),
                                     (BF_MIX, 300), (BF_DS, 8), (BF_DS, 64), (BF_DS, 257)],
                         ids=["f32-T7", "f32-T100", "mix-T1", "mix-T16", "mix-T300", "ds-T8",
                              "ds-T64", "ds-T257"])
@pytest.mark.parametrize("rank", [8, 16])
def test_lora_forward_parity(shape, T, rank):
    tol = TOL_F32 if shape.dtype == I.F32 else TOL_BF16
    y, ref, base = _case(shape, T, rank, 60 + T, lambda e: e % 3 != 1)  # some experts unadapted
    check_output(y, ref, tol, f"{shape.name} T={T} r={rank}")
    # the adapters change the output well beyond the tolerance (the test would see them missing)
    row, _ = oracle.ffn.rel_err_rows(base, ref)
    assert row.max() > 5 * tol


def test_lora_rejects_bad_rank():
    sh = BF_MIX
    desc = M.desc_of(sh)
    with pytest.raises(M.MCFTError) as ei:
        M.mcft_moe_workspace_size_lora(desc, 4, 16)
    assert ei.value.status == M.MCFT_ERR_UNSUPPORTED


@pytest.mark.parametrize("shape,T", [(I.MIXTRAL, 16), (I.DSV2_LITE, 64), (I.MIXTRAL, 4096),
                                     (I.DSV2_LITE, 4096)],
                         ids=["mixtral-b16", "deepseek-b64", "mixtral-T4096", "deepseek-T4096"])
def test_lora_full_size(shape, T):
    """Full-size layers in Stage 2 (Section 3.2): routing restricted to a concentration set of 75 %
    of the experts (compact ratio r = 75 %, Section 4), rank-8 adapters (alpha 16, Appendix B) on
    the experts of the set and on the shared experts. Every row is compared with the oracle, at
    the decode batches and at T = 4096 (tcgen05 path, the size the bench times)."""
    seed = 70 + T
    lw = weights(shape)
    kept = [int(e) for e in np.nonzero(I.keep_mask(seed, shape.E, shape.E * 3 // 4))[0]]
    ids = I.random_ids(seed, 1, T, shape.K, shape.E, hot=kept, p_hot=1.0)[0]
    assert np.isin(ids, kept).all()
    gate = np.random.default_rng(seed).uniform(0.05, 1.0, (T, shape.K)).astype(np.float32)
    x = I.hidden_iid(seed, shape, T)
    ad = [I.lora_block(seed, shape, e, 8) if e in kept else None for e in range(shape.E)]
    sad = [I.lora_block(seed, shape, ("shared", s), 8) for s in range(shape.n_shared)]
    desc = M.desc_of(shape)
    y = M.mcft_moe_forward_lora(
        desc, x.to(DEV), torch.from_numpy(ids).to(DEV), torch.from_numpy(gate).to(DEV),
        [lw.experts[e].to(DEV) if e in kept else None for e in range(shape.E)],
        [b.to(DEV) for b in lw.shared], [None if b is None else b.to(DEV) for b in ad],
        [b.to(DEV) for b in sad], 8, 2.0)
    M.mcft_device_error()
    assert torch.isfinite(y.float()).all()
    split = lambda b: None if b is None else tuple(f64(t) for t in I.split_lora(b, shape, 8))
    ex = [tuple(f64(t) for t in I.split_expert(lw.experts[e], shape)) if e in kept else None
          for e in range(shape.E)]
    ref = oracle.ffn.moe_layer(f64(x), ids, gate.astype(np.float64), ex, shared_triples(lw, shape),
                               lora=[split(b) for b in ad], shared_lora=[split(b) for b in sad],
                               lora_scale=2.0)
    check_output(y, ref, TOL_BF16, f"{shape.name} T={T} lora, every row")


@pytest.mark.parametrize("shape,T", [(I.MIXTRAL, 4096), (I.DSV2_LITE, 4096), (I.DSV2_LITE, 64),
                                     (BF_MIX, 300)],
                         ids=["mixtral-T4096", "deepseek-T4096", "deepseek-b64", "small-T300"])
@pytest.mark.parametrize("kind", ["zero-B", "no-adapter"])
def test_lora_without_effect_equals_plain_forward_bitwise(shape, T, kind):
    """Adapters whose up matrices are zero, or no adapter on any expert, add exact zeros: the
    Stage-2 forward then equals the plain forward bit for bit. On the tcgen05 path this runs the
    down projections, the builder warp's extra k-blocks and their hand-off, all adding 0."""
    seed = 90 + T
    lw = weights(shape)
    kept = [int(e) for e in np.nonzero(I.keep_mask(seed, shape.E, shape.E * 3 // 4))[0]]
    ids = I.random_ids(seed, 1, T, shape.K, shape.E, hot=kept, p_hot=1.0)[0]
    gate = np.random.default_rng(seed).uniform(0.05, 1.0, (T, shape.K)).astype(np.float32)
    x = I.hidden_iid(seed, shape, T).to(DEV)
    idx, g = torch.from_numpy(ids).to(DEV), torch.from_numpy(gate).to(DEV)
    experts = [lw.experts[e].to(DEV) if e in kept else None for e in range(shape.E)]
    shared = [b.to(DEV) for b in lw.shared]

    def zero_b(b):
        b = b.clone()
        for t, part in zip(I.split_lora(b, shape, 8), range(6)):
            if part % 2 == 1:  # B1, B3, B2
                t.zero_()
        return b.to(DEV)

    if kind == "zero-B":
        ad = [zero_b(I.lora_block(seed, shape, e, 8)) if e in kept else None for e in range(shape.E)]
        sad = [zero_b(I.lora_block(seed, shape, ("shared", s), 8)) for s in range(shape.n_shared)]
    else:
        ad = [None] * shape.E
        sad = [None] * shape.n_shared
    desc = M.desc_of(shape)
    y_l = M.mcft_moe_forward_lora(desc, x, idx, g, experts, shared, ad, sad, 8, 2.0)
    y_p = M.mcft_moe_forward(desc, x, idx, g, experts, shared)
    M.mcft_device_error()
    assert torch.equal(y_l, y_p), f"{shape.name} T={T} {kind}"
