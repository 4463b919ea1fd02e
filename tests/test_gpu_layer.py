"""End-to-end decode steps through the C ABI: route (soft prior) -> cache step -> fetch of missed
experts from pinned host memory -> expert FFN + combine, against the oracle's routing, cache and
layer output (Section 3.1, Eq. inference, Section 4.1). Two fetch paths: the host reads the miss
list and issues copies (mcft_fetch_experts + mcft_moe_forward), or the device copies the missed
experts itself while the hit experts are computed (mcft_moe_forward_cached)."""
import numpy as np
import pytest
import torch

import oracle
from paper_2609_34077_gb300 import inputs as I
from paper_2609_34077_gb300 import mcft as M
from tests.gpu_helpers import NEAR_TIE, TOL_BF16, check_output, expert_triples, f64, shared_triples

pytestmark = pytest.mark.gpu
DEV = "cuda"

SMALL_MIX = I.LayerShape("small-mix", d=256, E=8, K=2, w=256, n_shared=0, gate=I.GATE_RENORM,
                         dtype=I.BF16, cache_slots=4, keep=4)
SMALL_DS = I.LayerShape("small-ds-layer", d=256, E=64, K=6, w=128, n_shared=2, gate=I.GATE_PLAIN,
                        dtype=I.BF16, cache_slots=12, keep=16)


def _decode_stream(shape, batch, steps, seed, check_every=1, path="host", policy="LRU"):
    lw = I.layer_weights(seed, shape, pin=True)
    desc = M.desc_of(shape)
    prior = I.prior_from_mask(I.keep_mask(seed, shape.E, shape.keep))
    xs = I.ar1_streams(seed, shape, steps, batch)
    cache = M.mcft_cache_create(1, shape.E, shape.cache_slots, shape.expert_bytes, lw.experts,
                                max_assign=batch * shape.K, policy=policy)
    ref_cache = oracle.cache.SlotCache(shape.E, shape.cache_slots, policy)
    wr = lw.router.to(DEV)
    shared = [b.to(DEV) for b in lw.shared]
    ws = torch.empty(M.mcft_moe_workspace_size(desc, batch), dtype=torch.uint8, device=DEV)
    copy = torch.cuda.Stream()
    ex_ref = expert_triples(lw, shape)
    sh_ref = shared_triples(lw, shape)
    mism = 0
    diverged = False  # once routing differs (a near tie), the two caches see different streams
    for s in range(steps):
        x = xs[s]
        xd = x.to(DEV)
        idx, gate = M.mcft_route(desc, xd, wr, M.MCFT_ROUTE_SOFT_PRIOR, prior=prior)
        M.mcft_cache_step(cache, 0, idx)
        if path == "host":
            ptrs = M.mcft_fetch_experts(cache, 0, torch.cuda.current_stream(), copy)
            y = M.mcft_moe_forward(desc, xd, idx, gate, ptrs, shared, workspace=ws)
        else:
            y = M.mcft_moe_forward_cached(desc, xd, idx, gate, cache, 0, shared, workspace=ws,
                                          copy_stream=copy)
            torch.cuda.synchronize()
        ref = oracle.routing.route(f64(x), f64(lw.router), shape.K, M.MCFT_ROUTE_SOFT_PRIOR,
                                   shape.gate, prior=prior)
        gi = idx.cpu().numpy()
        rows = np.all(gi == ref["idx"], axis=1)
        if not rows.all():
            near = (ref["gap_k"] < NEAR_TIE) | (ref["gap_in"] < NEAR_TIE)
            assert np.all(near[~rows]), f"step {s}: routing differs outside a near tie"
            mism += 1
            diverged = True
        h, f, b, ml = ref_cache.step(ref["idx"])
        if not diverged:
            assert M.mcft_cache_last_misses(cache, 0) == ml, f"step {s}"
        if s % check_every == 0 and rows.any():
            yref = oracle.ffn.moe_layer(f64(x)[rows], ref["idx"][rows], ref["gate"][rows], ex_ref, sh_ref)
            check_output(y[torch.from_numpy(np.nonzero(rows)[0]).to(DEV)], yref, TOL_BF16,
                         f"{shape.name} step {s}")
    M.mcft_device_error()
    return cache, mism


@pytest.mark.parametrize("path", ["host", "device"])
@pytest.mark.parametrize("shape,batch", [(SMALL_MIX, 1), (SMALL_MIX, 16), (SMALL_DS, 1),
                                         (SMALL_DS, 8), (SMALL_DS, 64)],
                         ids=["mix-b1", "mix-b16", "ds-b1", "ds-b8", "ds-b64"])
def test_decode_stream_small(shape, batch, path):
    _, mism = _decode_stream(shape, batch, 64, seed=20 + batch, path=path)
    assert mism <= 2


@pytest.mark.parametrize("policy", ["LFU", "FIFO"])
def test_decode_stream_policies_device_fetch(policy):
    _, mism = _decode_stream(SMALL_DS, 8, 48, seed=27, path="device", policy=policy)
    assert mism <= 2


@pytest.mark.parametrize("path", ["host", "device"])
def test_decode_stream_mixtral_full_size(path):
    """Mixtral-shaped layer, 8 experts of 352 MB in pinned host memory, 4 GPU slots: 12 decode
    steps at batch 1 with real fetches; output checked every 4th step."""
    _, mism = _decode_stream(I.MIXTRAL, 1, 12, seed=30, check_every=4, path=path)
    assert mism <= 1


def test_forward_cached_rejects_prefill_and_accounting_caches():
    sh = SMALL_MIX
    desc = M.desc_of(sh)
    acc = M.mcft_cache_create(1, sh.E, sh.cache_slots, max_assign=2)
    x = torch.zeros((1, sh.d), dtype=torch.bfloat16, device=DEV)
    idx = torch.zeros((1, 2), dtype=torch.int32, device=DEV)
    idx[0, 1] = 1
    g = torch.ones((1, 2), device=DEV)
    with pytest.raises(M.MCFTError):
        M.mcft_moe_forward_cached(desc, x, idx, g, acc, 0)


@pytest.mark.parametrize("shape,T", [(SMALL_DS, 1), (SMALL_DS, 5), (SMALL_DS, 40), (SMALL_MIX, 16)],
                         ids=["ds-b1", "ds-b5", "ds-b40", "mix-b16"])
def test_cached_forward_equals_plain_forward_bitwise(shape, T):
    """Where an expert's bytes come from does not change the bf16 decode output: a hit (first FFN
    phase), a demand fetch or bypass (second phase), a prefetch still landing (second phase) and a
    resident expert of the plain forward give the same bits, because the decode work items have
    the same shape and summation order in every launch of a layer and batch size."""
    desc = M.desc_of(shape)
    lw = I.layer_weights(80, shape, pin=True)
    cache = M.mcft_cache_create(1, shape.E, shape.cache_slots, shape.expert_bytes, lw.experts,
                                max_assign=T * shape.K)
    experts = [b.to(DEV) for b in lw.experts]
    shared = [b.to(DEV) for b in lw.shared]
    compute, copy = torch.cuda.Stream(), torch.cuda.Stream()
    steps = 8
    ids = I.random_ids(80, steps, T, shape.K, shape.E, hot=range(shape.keep), p_hot=0.8)
    gates = np.random.default_rng(80).uniform(0.05, 1.0, (steps, T, shape.K)).astype(np.float32)
    xs = [I.hidden_iid(81 + s, shape, T).to(DEV) for s in range(steps)]
    idxs = [torch.from_numpy(ids[s]).to(DEV) for s in range(steps)]
    gts = [torch.from_numpy(gates[s]).to(DEV) for s in range(steps)]
    wsz = M.mcft_moe_workspace_size(desc, T)
    ws_c, ws_p = (torch.empty(wsz, dtype=torch.uint8, device=DEV) for _ in range(2))
    y_c, y_p = (torch.empty((T, shape.d), dtype=torch.bfloat16, device=DEV) for _ in range(2))
    torch.cuda.synchronize()
    for s in range(steps):
        M.mcft_cache_step(cache, 0, idxs[s], stream=compute)
        M.mcft_moe_forward_cached(desc, xs[s], idxs[s], gts[s], cache, 0, shared, y=y_c,
                                  workspace=ws_c, compute_stream=compute, copy_stream=copy)
        if s % 2 == 0 and s + 1 < steps:  # the next step then finds some experts still landing
            M.mcft_cache_prefetch(cache, 0, idxs[s + 1], min(2, shape.cache_slots), stream=compute)
        M.mcft_moe_forward(desc, xs[s], idxs[s], gts[s], experts, shared, y=y_p, workspace=ws_p,
                           stream=compute)
        compute.synchronize()
        copy.synchronize()
        assert torch.equal(y_c, y_p), f"step {s}"
    M.mcft_device_error()
    assert M.mcft_cache_stats(cache, 0)[1] > 0  # the stream did fetch


def _prefill_full(shape, keep, seed):
    """The masked fine-tuning / prefill forward at full size: T = 4096 tokens routed by mcft_route
    under a hard mask keeping `keep` experts, then mcft_moe_forward (tcgen05 grouped GEMMs),
    against the oracle on every one of the 4096 rows."""
    T = 4096
    mask = I.keep_mask(seed, shape.E, keep)
    kept = [int(e) for e in np.nonzero(mask)[0]]
    lw = I.layer_weights(seed, shape, experts=kept)
    desc = M.desc_of(shape)
    x = I.hidden_iid(seed, shape, T)
    xd = x.to(DEV)
    idx, gate = M.mcft_route(desc, xd, lw.router.to(DEV), M.MCFT_ROUTE_HARD_MASK, mask=mask)
    y = M.mcft_moe_forward(desc, xd, idx, gate, [None if b is None else b.to(DEV) for b in lw.experts],
                           [b.to(DEV) for b in lw.shared])
    M.mcft_device_error()
    ref = oracle.routing.route(f64(x), f64(lw.router), shape.K, M.MCFT_ROUTE_HARD_MASK, shape.gate,
                               mask=mask)
    from tests.gpu_helpers import check_routing

    flagged, _ = check_routing(idx, gate, ref, shape.gate)
    assert flagged < T // 100
    gi = idx.cpu().numpy()
    assert np.all(mask[gi] == 1)
    # the layer for the experts the GPU chose (the oracle's own set outside near ties), with the
    # oracle's gates for them (from its p)
    pa = np.take_along_axis(ref["p"], gi.astype(np.int64), axis=1)
    g_ref = pa / pa.sum(axis=1, keepdims=True) if shape.gate == I.GATE_RENORM else pa
    yref = oracle.ffn.moe_layer(f64(x), gi, g_ref, expert_triples(lw, shape), shared_triples(lw, shape))
    row, fro = check_output(y, yref, TOL_BF16, f"{shape.name} prefill T={T}, every row")
    assert fro < TOL_BF16
    return row, fro


def test_prefill_mixtral_full_size_every_row():
    """Mixtral-shaped, T = 8 x 512 = 4096, hard mask keeping 4 of 8 experts (unbalanced loads:
    8192 assignments over the 4 kept experts, each padded to 128-row tiles)."""
    _prefill_full(I.MIXTRAL, 4, seed=90)


def test_prefill_deepseek_full_size_every_row():
    """DeepSeek-V2-Lite-shaped, T = 4096, 64 routed experts (hard mask keeping 48) plus the 2
    shared experts on every token: 24576 routed and 8192 shared rows through the grouped GEMMs."""
    _prefill_full(I.DSV2_LITE, 48, seed=91)


@pytest.mark.parametrize("T,fetching", [(1, "ffn_decode_fetch"), (16, "ffn_decode_fetch"),
                                        (17, "fetch"), (40, "fetch")])
def test_cached_forward_fetches_in_the_ffn_launch_up_to_16_tokens(T, fetching):
    """Which launch moves the misses: up to 16 tokens (with no prefetch in flight) the decode FFN
    launch itself, above that the fetch kernel on the copy stream beside a two-phase FFN."""
    shape = SMALL_DS
    desc = M.desc_of(shape)
    lw = I.layer_weights(85, shape, pin=True)
    cache = M.mcft_cache_create(1, shape.E, shape.cache_slots, shape.expert_bytes, lw.experts,
                                max_assign=T * shape.K)
    shared = [b.to(DEV) for b in lw.shared]
    x = I.hidden_iid(86, shape, T).to(DEV)
    idx = torch.from_numpy(I.random_ids(85, 1, T, shape.K, shape.E, hot=range(shape.keep))[0]).to(DEV)
    gate = torch.full((T, shape.K), 0.2, device=DEV)
    torch.cuda.synchronize()
    M.mcft_profile_reset()
    M.mcft_profile_enable(True)
    M.mcft_cache_step(cache, 0, idx)
    M.mcft_moe_forward_cached(desc, x, idx, gate, cache, 0, shared, copy_stream=torch.cuda.Stream())
    M.mcft_profile_enable(False)
    prof = {k: v[0] for k, v in M.mcft_profile_read().items() if v[0]}
    M.mcft_device_error()
    assert prof.get(fetching, 0) == 1, prof
    other = "fetch" if fetching == "ffn_decode_fetch" else "ffn_decode_fetch"
    assert prof.get(other, 0) == 0, prof
    assert prof.get("ffn_decode", 0) == (0 if fetching == "ffn_decode_fetch" else 2), prof
