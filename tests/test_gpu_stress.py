"""Randomised decode streams through the device-driven cached forward: random bf16 layer shapes
(8, 16 or 64 routed experts, K up to 6, up to 2 shared experts), batch sizes 1-48, cache budgets,
replacement policies and prefetch settings, many steps each. At every step the cached forward (hit
experts in its first FFN phase; demand fetches, bypasses and prefetches still landing in its second,
next to the fetch kernel) must equal the plain forward with every expert resident, bit for bit,
and the cache's miss list must equal the oracle cache's (Section 4.1 "Simulation"). The
claimed-item FFN with its GEMM13 -> GEMM2 waits, the fetch kernel's reserved slots and the prefetch
cancel path all run many times here."""
import numpy as np
import pytest
import torch

import oracle
from paper_2609_34077_gb300 import inputs as I
from paper_2609_34077_gb300 import mcft as M

pytestmark = pytest.mark.gpu
DEV = "cuda"


def _shape(rng, i):
    E = int(rng.choice([8, 16, 64]))
    K = int(rng.integers(1, min(6, E // 2) + 1))
    B = int(rng.integers(K, E))  # K <= B < E
    return I.LayerShape(f"stress-{i}", d=int(rng.choice([128, 256, 512])), E=E, K=K,
                        w=int(rng.choice([64, 128, 192, 384])), n_shared=int(rng.integers(0, 3)),
                        gate=I.GATE_RENORM if rng.random() < 0.5 else I.GATE_PLAIN, dtype=I.BF16,
                        cache_slots=B, keep=min(E, B + 2))


@pytest.mark.parametrize("seed", range(24))
def test_random_decode_streams_cached_equals_plain(seed):
    rng = np.random.default_rng(1000 + seed)
    shape = _shape(rng, seed)
    T = int(rng.choice([1, 2, 5, 16, 33, 48]))
    policy = str(rng.choice(["LRU", "LFU", "FIFO"]))
    n_pf = int(rng.integers(0, min(3, shape.cache_slots) + 1))
    steps = 32
    desc = M.desc_of(shape)
    lw = I.layer_weights(2000 + seed, shape, pin=True)
    cache = M.mcft_cache_create(1, shape.E, shape.cache_slots, shape.expert_bytes, lw.experts,
                                max_assign=T * shape.K, policy=policy)
    ref = oracle.cache.SlotCache(shape.E, shape.cache_slots, policy)
    experts = [b.to(DEV) for b in lw.experts]
    shared = [b.to(DEV) for b in lw.shared]
    hot = range(shape.keep)
    ids = I.random_ids(3000 + seed, steps, T, shape.K, shape.E, hot=hot, p_hot=0.7)
    preds = I.random_ids(4000 + seed, steps, T, shape.K, shape.E, hot=hot, p_hot=0.7)
    gates = rng.uniform(0.05, 1.0, (steps, T, shape.K)).astype(np.float32)
    xs = [I.hidden_iid(5000 + 100 * seed + s, shape, T).to(DEV) for s in range(steps)]
    idxs = [torch.from_numpy(ids[s]).to(DEV) for s in range(steps)]
    pdev = [torch.from_numpy(preds[s]).to(DEV) for s in range(steps)]
    gts = [torch.from_numpy(gates[s]).to(DEV) for s in range(steps)]
    wsz = M.mcft_moe_workspace_size(desc, T)
    ws_c, ws_p = (torch.empty(wsz, dtype=torch.uint8, device=DEV) for _ in range(2))
    y_c, y_p = (torch.empty((T, shape.d), dtype=torch.bfloat16, device=DEV) for _ in range(2))
    compute, copy = torch.cuda.Stream(), torch.cuda.Stream()
    torch.cuda.synchronize()
    what = f"{shape} T={T} {policy} prefetch={n_pf}"
    fetched = 0
    for s in range(steps):
        M.mcft_cache_step(cache, 0, idxs[s], stream=compute)
        _, f, _, ml = ref.step(ids[s])
        fetched += f
        M.mcft_moe_forward_cached(desc, xs[s], idxs[s], gts[s], cache, 0, shared, y=y_c,
                                  workspace=ws_c, compute_stream=compute, copy_stream=copy)
        if n_pf and s % 2 == 0 and s + 1 < steps:  # the next step finds some experts landing
            M.mcft_cache_prefetch(cache, 0, pdev[s], n_pf, stream=compute)
            ref.prefetch(oracle.stack.prefetch_candidates(preds[s]), n_pf)
        M.mcft_moe_forward(desc, xs[s], idxs[s], gts[s], experts, shared, y=y_p, workspace=ws_p,
                           stream=compute)
        compute.synchronize()
        copy.synchronize()
        assert M.mcft_cache_last_misses(cache, 0) == ml, f"{what} step {s}"
        assert torch.equal(y_c, y_p), f"{what} step {s}"
    M.mcft_device_error()
    assert M.mcft_cache_stats(cache, 0)[1] == fetched > 0
