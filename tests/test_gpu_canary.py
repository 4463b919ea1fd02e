"""Out-of-bounds writes: every output and workspace buffer sits between guard regions of a known byte
pattern, and after each call the guards must be untouched. This stands in for a memory sanitizer
(closed on this pool) for the library's writes: the routing outputs, the forward's workspace and
output on every FFN path (tensor-core prefill, bf16 decode at each batch class, fp32 rowwise,
LoRA, the device-driven cached forward), the residual/RMSNorm kernel and a chained-stack step.
The last element before each guard is exactly the end of the buffer, so a write one element past
the end is caught."""
import numpy as np
import pytest
import torch

from paper_2609_34077_gb300 import inputs as I
from paper_2609_34077_gb300 import mcft as M

pytestmark = pytest.mark.gpu
DEV = "cuda"
GUARD = 4096  # bytes on each side (a multiple of 256 keeps every buffer's alignment)
PATTERN = 0xA5

SMALL_BF16 = I.LayerShape("canary-bf16", d=512, E=8, K=2, w=384, n_shared=0, gate=I.GATE_RENORM,
                          dtype=I.BF16, cache_slots=4, keep=4)
SMALL_DS = I.LayerShape("canary-ds", d=256, E=64, K=6, w=128, n_shared=2, gate=I.GATE_PLAIN,
                        dtype=I.BF16, cache_slots=12, keep=16)


class Guarded:
    """A device buffer of `nbytes` between two guard regions; view(dtype, shape) gives the buffer."""

    def __init__(self, nbytes):
        self.n = int(nbytes)
        self.raw = torch.full((GUARD + self.n + GUARD,), PATTERN, dtype=torch.uint8, device=DEV)

    def view(self, dtype=torch.uint8, shape=None):
        v = self.raw[GUARD:GUARD + self.n].view(dtype)
        return v if shape is None else v.view(shape)

    def check(self, what):
        torch.cuda.synchronize()
        lo = self.raw[:GUARD]
        hi = self.raw[GUARD + self.n:]
        assert bool((lo == PATTERN).all()), f"{what}: write before the buffer"
        assert bool((hi == PATTERN).all()), f"{what}: write past the end of the buffer"


def _tdtype(shape):
    return torch.bfloat16 if shape.dtype == I.BF16 else torch.float32


def _esize(shape):
    return 2 if shape.dtype == I.BF16 else 4


def _ids(shape, T, seed):
    ids = I.random_ids(seed, 1, T, shape.K, shape.E, hot=range(shape.keep), p_hot=0.8)[0]
    gate = np.random.default_rng(seed).uniform(0.05, 1.0, (T, shape.K)).astype(np.float32)
    return torch.from_numpy(ids).to(DEV), torch.from_numpy(gate).to(DEV)


@pytest.mark.parametrize("shape,T", [(I.TINY, 1), (I.TINY, 37), (SMALL_BF16, 1), (SMALL_BF16, 16),
                                     (SMALL_BF16, 64), (SMALL_BF16, 300), (SMALL_DS, 5),
                                     (SMALL_DS, 130)],
                         ids=lambda v: getattr(v, "name", str(v)))
def test_route_and_forward_stay_in_bounds(shape, T):
    desc = M.desc_of(shape)
    lw = I.layer_weights(70, shape)
    x = I.hidden_iid(70, shape, T).to(DEV)
    experts = [b.to(DEV) for b in lw.experts]
    shared = [b.to(DEV) for b in lw.shared]
    gidx, ggate = Guarded(T * shape.K * 4), Guarded(T * shape.K * 4)
    idx, gate = gidx.view(torch.int32, (T, shape.K)), ggate.view(torch.float32, (T, shape.K))
    prior = I.prior_from_mask(I.keep_mask(70, shape.E, shape.keep))
    M.mcft_route(desc, x, lw.router.to(DEV), M.MCFT_ROUTE_SOFT_PRIOR, prior=prior, idx=idx, gate=gate)
    gidx.check("route idx")
    ggate.check("route gate")
    gws = Guarded(M.mcft_moe_workspace_size(desc, T))
    gy = Guarded(T * shape.d * _esize(shape))
    y = gy.view(_tdtype(shape), (T, shape.d))
    M.mcft_moe_forward(desc, x, idx, gate, experts, shared, y=y, workspace=gws.view())
    M.mcft_device_error()
    gws.check("forward workspace")
    gy.check("forward output")
    assert bool(torch.isfinite(y.float()).all())


@pytest.mark.parametrize("T", [1, 16, 300])
def test_lora_forward_stays_in_bounds(T):
    shape, rank = SMALL_BF16, 8
    desc = M.desc_of(shape)
    lw = I.layer_weights(71, shape)
    x = I.hidden_iid(71, shape, T).to(DEV)
    idx, gate = _ids(shape, T, 71)
    lora = [I.lora_block(71, shape, e, rank).to(DEV) for e in range(shape.E)]
    gws = Guarded(M.mcft_moe_workspace_size_lora(desc, rank, T))
    gy = Guarded(T * shape.d * 2)
    y = gy.view(torch.bfloat16, (T, shape.d))
    M.mcft_moe_forward_lora(desc, x, idx, gate, [b.to(DEV) for b in lw.experts], expert_lora=lora,
                            rank=rank, scale=2.0, y=y, workspace=gws.view())
    M.mcft_device_error()
    gws.check("LoRA workspace")
    gy.check("LoRA output")


@pytest.mark.parametrize("shape,T", [(SMALL_BF16, 1), (SMALL_BF16, 16), (SMALL_DS, 8)],
                         ids=lambda v: getattr(v, "name", str(v)))
def test_cached_forward_and_cache_stay_in_bounds(shape, T):
    desc = M.desc_of(shape)
    lw = I.layer_weights(72, shape, pin=True)
    cache = M.mcft_cache_create(1, shape.E, shape.cache_slots, shape.expert_bytes, lw.experts,
                                max_assign=T * shape.K)
    shared = [b.to(DEV) for b in lw.shared]
    gws = Guarded(M.mcft_moe_workspace_size(desc, T))
    gy = Guarded(T * shape.d * 2)
    y = gy.view(torch.bfloat16, (T, shape.d))
    compute, copy = torch.cuda.Stream(), torch.cuda.Stream()
    xs = [I.hidden_iid(72 + s, shape, T).to(DEV) for s in range(6)]
    ids = [_ids(shape, T, 72 + s) for s in range(6)]
    torch.cuda.synchronize()
    for s in range(6):
        idx, gate = ids[s]
        M.mcft_cache_step(cache, 0, idx, stream=compute)
        if s % 2:
            M.mcft_cache_prefetch(cache, 0, ids[(s + 1) % 6][0], min(2, shape.cache_slots),
                                  stream=compute)
        M.mcft_moe_forward_cached(desc, xs[s], idx, gate, cache, 0, shared, y=y,
                                  workspace=gws.view(), compute_stream=compute, copy_stream=copy)
    compute.synchronize()
    copy.synchronize()
    M.mcft_device_error()
    gws.check("cached forward workspace")
    gy.check("cached forward output")


@pytest.mark.parametrize("shape,T", [(I.TINY, 3), (SMALL_DS, 1), (I.MIXTRAL, 2)],
                         ids=lambda v: getattr(v, "name", str(v)))
def test_norm_stays_in_bounds(shape, T):
    desc = M.desc_of(shape)
    gx = Guarded(T * shape.d * 4)
    gu = Guarded(T * shape.d * _esize(shape))
    x = gx.view(torch.float32, (T, shape.d))
    x.copy_(torch.from_numpy(I.normal_f32(73, "canary-x", T * shape.d).reshape(T, shape.d)))
    y = I.hidden_iid(73, shape, T).to(DEV)
    u = gu.view(_tdtype(shape), (T, shape.d))
    M.mcft_residual_rmsnorm(desc, x, y, I.norm_weight(73, shape).to(DEV), eps=shape.norm_eps, u=u)
    gx.check("stream")
    gu.check("normalised input")


@pytest.mark.parametrize("T", [1, 4])
def test_stack_step_stays_in_bounds(T):
    """A 3-layer chained stack step (T = 1 runs the fused prologue) writes only its stream."""
    shape, L = SMALL_DS, 3
    desc = M.desc_of(shape)
    lws = [I.layer_weights(74, shape, layer=l, pin=True) for l in range(L)]
    cache = M.mcft_cache_create(L, shape.E, shape.cache_slots, shape.expert_bytes,
                                [lw.experts[e] for lw in lws for e in range(shape.E)],
                                max_assign=T * shape.K)
    priors = np.stack([I.prior_from_mask(I.keep_mask(74, shape.E, shape.keep, l)) for l in range(L)])
    stack = M.mcft_stack_create(desc, [lw.router.to(DEV) for lw in lws], priors,
                                [I.norm_weight(74, shape, l).to(DEV) for l in range(L)],
                                [[b.to(DEV) for b in lw.shared] for lw in lws], shape.norm_eps,
                                cache, n_prefetch=2, T_max=T)
    gx = Guarded(T * shape.d * 4)
    x = gx.view(torch.float32, (T, shape.d))
    for s in range(3):
        x.copy_(I.residual_stream(74, shape, 3, T)[s].to(DEV))
        M.mcft_stack_step(stack, x)
    M.mcft_device_error()
    gx.check("stack stream")
