"""Prefetch events of the device cache (mcft_cache_prefetch) against the oracle, bit-exact.

Decisions: random predicted routings and step routings through the device cache in accounting mode
and through oracle.cache.SlotCache with oracle.stack.prefetch_candidates; slot tags after every event and
all five counters must be equal. Data: with slots and pinned host blocks, every expert a step
selects must hold its host block's bytes, whether it came from the step's own fetch, from a
prefetch streamed in behind an earlier layer's misses, or from an earlier step."""
import numpy as np
import pytest
import torch

import oracle
from paper_2609_34077_gb300 import inputs as I
from paper_2609_34077_gb300 import mcft as M
from tests.gpu_helpers import device_view

pytestmark = pytest.mark.gpu
DEV = "cuda"


@pytest.mark.parametrize("policy", ["LRU", "LFU", "FIFO"])
@pytest.mark.parametrize("E,B,K,T,n_max", [(8, 4, 2, 1, 2), (8, 4, 2, 4, 3), (64, 12, 6, 1, 6),
                                           (64, 12, 6, 8, 12), (5, 2, 1, 3, 1)])
def test_prefetch_decisions_exact(policy, E, B, K, T, n_max):
    steps = 120
    hot = range(min(E, B + 3))
    ids = I.random_ids(21, steps, T, K, E, hot=hot, p_hot=0.7)
    preds = I.random_ids(22, steps, T, K, E, hot=hot, p_hot=0.7)
    c = M.mcft_cache_create(1, E, B, max_assign=T * K, policy=policy)
    ref = oracle.cache.SlotCache(E, B, policy)
    th = tf = tb = 0
    for s in range(steps):
        if s % 3 != 2:
            M.mcft_cache_prefetch(c, 0, torch.from_numpy(preds[s]).to(DEV), n_max)
            ref.prefetch(oracle.stack.prefetch_candidates(preds[s]), n_max)
            assert M.mcft_cache_tags(c, 0) == ref.tag, f"after the prefetch before step {s}"
        M.mcft_cache_step(c, 0, torch.from_numpy(ids[s]).to(DEV))
        h, f, b, _ = ref.step(ids[s])
        th, tf, tb = th + h, tf + f, tb + b
        assert M.mcft_cache_tags(c, 0) == ref.tag, f"after step {s}"
    assert M.mcft_cache_stats(c, 0) == (th, tf, tb)
    assert M.mcft_cache_prefetch_stats(c, 0)[:2] == (ref.prefetched, ref.useful)
    assert ref.prefetched > 0 and ref.useful > 0


def test_prefetch_export_import_resume():
    """A checkpoint taken between steps carries the pending prefetch set (useful counts resume)."""
    E, B, K, steps, cut = 8, 4, 2, 60, 25
    ids = I.random_ids(23, steps, 1, K, E, hot=range(6), p_hot=0.7)
    preds = I.random_ids(24, steps, 1, K, E, hot=range(6), p_hot=0.7)

    def run(c, lo, hi):
        for s in range(lo, hi):
            M.mcft_cache_prefetch(c, 0, torch.from_numpy(preds[s]).to(DEV), 2)
            if s == hi - 1 and hi == cut:
                return  # stop right after a prefetch: its set is pending
            M.mcft_cache_step(c, 0, torch.from_numpy(ids[s]).to(DEV))

    a = M.mcft_cache_create(1, E, B, max_assign=K, policy="LRU")
    run(a, 0, cut)
    state = M.mcft_cache_export(a)
    b = M.mcft_cache_create(1, E, B, max_assign=K, policy="LRU")
    M.mcft_cache_import(b, state)
    for c in (a, b):
        M.mcft_cache_step(c, 0, torch.from_numpy(ids[cut - 1]).to(DEV))
        run(c, cut, steps)
    assert M.mcft_cache_stats(a, 0) == M.mcft_cache_stats(b, 0)
    assert M.mcft_cache_prefetch_stats(a, 0)[:2] == M.mcft_cache_prefetch_stats(b, 0)[:2]
    assert M.mcft_cache_tags(a, 0) == M.mcft_cache_tags(b, 0)


def test_prefetch_invalid():
    c = M.mcft_cache_create(2, 8, 4, max_assign=2)
    p = torch.zeros((1, 2), dtype=torch.int32, device=DEV)
    for n_max in (0, 5):
        with pytest.raises(M.MCFTError):
            M.mcft_cache_prefetch(c, 0, p, n_max)
    with pytest.raises(M.MCFTError):
        M.mcft_cache_prefetch(c, 2, p, 2)
    with pytest.raises(M.MCFTError):  # T*K > max_assign
        M.mcft_cache_prefetch(c, 0, torch.zeros((2, 2), dtype=torch.int32, device=DEV), 2)


def test_prefetched_bytes_land_in_the_right_slots():
    """Three layers of random byte blocks: per step, layer l's cache step, then the prefetch of
    layer l+1 from a random prediction, then mcft_fetch_experts of layer l (which streams layer
    l+1's prefetch in behind layer l's misses). After each step every selected expert's address
    holds its host block."""
    L, E, B, K, nbytes = 3, 8, 3, 2, 1 << 20
    g = torch.Generator().manual_seed(25)
    host = [torch.randint(0, 256, (nbytes,), dtype=torch.uint8, generator=g).pin_memory()
            for _ in range(L * E)]
    c = M.mcft_cache_create(L, E, B, nbytes, host, max_assign=K, policy="LRU")
    steps = 40
    ids = I.random_ids(26, steps * L, 1, K, E, hot=range(5), p_hot=0.7).reshape(steps, L, 1, K)
    preds = I.random_ids(27, steps * L, 1, K, E, hot=range(5), p_hot=0.7).reshape(steps, L, 1, K)
    compute, copy = torch.cuda.Stream(), torch.cuda.Stream()
    ids_d, preds_d = torch.from_numpy(ids).to(DEV), torch.from_numpy(preds).to(DEV)
    torch.cuda.synchronize()  # inputs are ready before the other streams read them
    checked = 0
    for s in range(steps):
        ptrs = []
        for l in range(L):
            M.mcft_cache_step(c, l, ids_d[s, l], stream=compute)
            if l + 1 < L:
                M.mcft_cache_prefetch(c, l + 1, preds_d[s, l + 1], 2, stream=compute)
            ptrs.append(M.mcft_fetch_experts(c, l, compute, copy))
        compute.synchronize()
        copy.synchronize()
        for l in range(L):
            for e in np.unique(ids[s, l]):
                got = device_view(ptrs[l][e], nbytes, torch.uint8).cpu()
                assert torch.equal(got, host[l * E + int(e)]), f"step {s} layer {l} expert {e}"
                checked += 1
    M.mcft_device_error()
    p, u, moved = M.mcft_cache_prefetch_stats(c)
    assert p > 0 and u > 0
    assert 0 < moved <= p * nbytes  # dropped prefetches may stop early
    assert checked == sum(len(np.unique(ids[s, l])) for s in range(steps) for l in range(L))


def test_prefetch_with_the_device_driven_forward():
    """The same pattern through mcft_moe_forward_cached on tiny fp32 layers: the outputs must equal
    the oracle's layer on the same routing (every expert the FFN reads came through a slot)."""
    shape = I.TINY
    L, E, B, K = 3, shape.E, 3, shape.K
    desc = M.desc_of(shape)
    lws = [I.layer_weights(28, shape, layer=l, pin=True) for l in range(L)]
    host = [lw.experts[e] for lw in lws for e in range(E)]
    triples = [[tuple(t.double().numpy() for t in I.split_expert(b, shape)) for b in lw.experts]
               for lw in lws]
    c = M.mcft_cache_create(L, E, B, shape.expert_bytes, host, max_assign=K, policy="LFU")
    steps = 24
    ids = I.random_ids(29, steps * L, 1, K, E, hot=range(5), p_hot=0.7).reshape(steps, L, 1, K)
    preds = I.random_ids(30, steps * L, 1, K, E, hot=range(5), p_hot=0.7).reshape(steps, L, 1, K)
    xs = I.hidden_iid(31, shape, steps * L).reshape(steps, L, 1, shape.d)
    gate = torch.tensor([[0.75, 0.25]], device=DEV)
    compute, copy = torch.cuda.Stream(), torch.cuda.Stream()
    ws = torch.empty(M.mcft_moe_workspace_size(desc, 1), dtype=torch.uint8, device=DEV)
    ys = torch.empty((steps, L, 1, shape.d), device=DEV)
    ids_d, preds_d, xs_d = (torch.from_numpy(ids).to(DEV), torch.from_numpy(preds).to(DEV),
                            xs.to(DEV))
    torch.cuda.synchronize()  # inputs are ready before the other streams read them
    for s in range(steps):
        for l in range(L):
            M.mcft_cache_step(c, l, ids_d[s, l], stream=compute)
            if l + 1 < L:
                M.mcft_cache_prefetch(c, l + 1, preds_d[s, l + 1], 2, stream=compute)
            M.mcft_moe_forward_cached(desc, xs_d[s, l], ids_d[s, l], gate, c, l, y=ys[s, l],
                                      workspace=ws, compute_stream=compute, copy_stream=copy)
    compute.synchronize()
    M.mcft_device_error()
    g = np.array([[0.75, 0.25]])
    for s in range(steps):
        for l in range(L):
            ref = oracle.ffn.moe_layer(xs[s, l].double().numpy(), ids[s, l], g, triples[l])
            got = ys[s, l].cpu().double().numpy()
            err = np.abs(got - ref).max() / np.abs(ref).max()
            assert err <= 1e-4, f"step {s} layer {l}: {err}"
    p, u, moved = M.mcft_cache_prefetch_stats(c)
    assert p > 0 and u > 0 and 0 < moved <= p * shape.expert_bytes
