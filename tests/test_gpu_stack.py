"""Full decode stacks, batch 1, 1024 steps: 32 Mixtral-shaped layers (B = 4) and 26 DeepSeek-
V2-Lite-shaped layers (B = 12), each layer with its own router, its own random soft-prior mask and
its own AR(1) hidden-state stream (layers are not chained). Routing runs on the GPU through
mcft_route and every (layer, step) goes through the device cache in accounting mode under LRU,
LFU and FIFO; per-layer hit and fetch counts, and Fetches/tok of Eq. metrics, must equal the
oracle's exactly (Section 4.1 "Simulation")."""
import numpy as np
import pytest

import oracle
from paper_2609_34077_gb300 import inputs as I
from paper_2609_34077_gb300 import mcft as M
from tests.gpu_helpers import NEAR_TIE, f64

pytestmark = pytest.mark.gpu
DEV = "cuda"
STEPS = 1024
POLICIES = ("LRU", "LFU", "FIFO")


@pytest.mark.parametrize("shape,L,B", [(I.MIXTRAL, 32, 4), (I.DSV2_LITE, 26, 12),
                                       (I.MIXTRAL, 32, 2), (I.MIXTRAL, 32, 6),
                                       (I.DSV2_LITE, 26, 24), (I.DSV2_LITE, 26, 36)],
                         ids=["mixtral-32-B4", "dsv2-26-B12", "mixtral-32-B2", "mixtral-32-B6",
                              "dsv2-26-B24", "dsv2-26-B36"])
def test_stack_fetch_counts_exact(shape, L, B):
    """Also the cache-budget sweep of Fig. 3 (B in {2, 4, 6} Mixtral, {12, 24, 36} DeepSeek)."""
    seed = 50
    desc = M.desc_of(shape)
    caches = {p: M.mcft_cache_create(L, shape.E, B, max_assign=shape.K, policy=p) for p in POLICIES}
    ref_counts = {p: np.zeros((L, 2), np.int64) for p in POLICIES}  # oracle (hits, fetches)
    exact_layers = []
    for layer in range(L):
        wr = I.router_weight(seed, shape, layer)
        prior = I.prior_from_mask(I.keep_mask(seed, shape.E, shape.keep, layer))
        x = I.ar1_streams(seed, shape, STEPS, 1, layer)[:, 0]
        idx, _ = M.mcft_route(desc, x.to(DEV), wr.to(DEV), M.MCFT_ROUTE_SOFT_PRIOR, prior=prior)
        r = oracle.routing.route(f64(x), f64(wr), shape.K, M.MCFT_ROUTE_SOFT_PRIOR, shape.gate,
                                 prior=prior)
        gi = idx.cpu().numpy()
        diff = np.any(gi != r["idx"], axis=1)
        if diff.any():
            near = (r["gap_k"] < NEAR_TIE) | (r["gap_in"] < NEAR_TIE)
            assert np.all(near[diff]), f"layer {layer}: routing differs outside a near tie"
        else:
            exact_layers.append(layer)
        for p in POLICIES:
            for s in range(STEPS):
                M.mcft_cache_step(caches[p], layer, idx[s:s + 1])
            oc = oracle.cache.SlotCache(shape.E, B, p)
            for s in range(STEPS):
                h, f, b, _ = oc.step(r["idx"][s])
                ref_counts[p][layer] += (h, f)
    M.mcft_device_error()
    assert len(exact_layers) >= L - 1  # at most one layer may hold a near tie that flips routing
    for p in POLICIES:
        tot = np.zeros(2, np.int64)
        for layer in exact_layers:
            h, f, b = M.mcft_cache_stats(caches[p], layer)
            assert b == 0
            assert (h, f) == tuple(ref_counts[p][layer]), f"{p} layer {layer}"
            tot += (h, f)
        n = len(exact_layers)
        hr, fpt = oracle.cache.metrics(tot[0], tot[1], STEPS, n, shape.K)
        assert fpt == pytest.approx(n * shape.K * (1 - hr))  # Eq. metrics at batch 1
        print(f"{shape.name} B={B} {p}: HR {100 * hr:.2f} %  Fetches/tok {fpt:.3f} over {n} layers")
