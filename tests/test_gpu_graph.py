"""A decode step of a multi-layer stack with the device-driven fetch has no host synchronisation,
so it can be captured as one CUDA graph and replayed per token. Replays must give the eager
outputs bit for bit (same kernels, same order) and leave the same cache state (Section 4.1)."""
import pytest
import torch

from paper_2609_34077_gb300 import inputs as I
from paper_2609_34077_gb300 import mcft as M

pytestmark = pytest.mark.gpu

SMALL = I.LayerShape("graph-ds", d=256, E=16, K=4, w=128, n_shared=2, gate=I.GATE_PLAIN,
                     dtype=I.BF16, cache_slots=6, keep=8)


@pytest.mark.parametrize("policy", ["LRU", "LFU"])
def test_graph_replay_equals_eager(policy):
    import bench

    dev = torch.device("cuda", 0)
    L, steps, warm = 4, 40, 6
    eager = bench.DecodeStack(SMALL, L, steps, 70, dev, policy)
    ys = []
    for s in range(steps):
        eager.step(s)
        torch.cuda.synchronize()
        ys.append(eager.y.clone())
    graphed = bench.DecodeStack(SMALL, L, steps, 70, dev, policy)
    for s in range(warm):
        graphed.step(s)
    torch.cuda.synchronize()
    graphed.capture()
    for s in range(warm, steps):
        graphed.step(s)
        torch.cuda.synchronize()
        assert torch.equal(graphed.y, ys[s]), f"step {s}"
    M.mcft_device_error()
    for l in range(L):
        assert M.mcft_cache_stats(graphed.cache, l) == M.mcft_cache_stats(eager.cache, l)
        assert M.mcft_cache_tags(graphed.cache, l) == M.mcft_cache_tags(eager.cache, l)
    h, f, b = M.mcft_cache_stats(graphed.cache, -1)
    assert f > 0 and h > 0  # the stream exercised both hits and device-driven fetches
