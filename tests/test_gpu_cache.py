"""GPU expert cache (device LRU decisions, counters, miss lists, fetches from pinned host memory)
against the oracle, through the C ABI. Section 4.1 "Simulation" and Eq. metrics; decisions and
counts must be bit-exact."""
import numpy as np
import pytest
import torch

import oracle
from paper_2609_34077_gb300 import inputs as I
from paper_2609_34077_gb300 import mcft as M
from tests.gpu_helpers import device_view

pytestmark = pytest.mark.gpu
DEV = "cuda"


def _stream_ids(E, K, T, steps, keep, seed):
    return I.random_ids(seed, steps, T, K, E, hot=range(keep), p_hot=0.75)


@pytest.mark.parametrize("policy", ["LRU", "LFU", "FIFO"])
@pytest.mark.parametrize("E,B,K,T", [(8, 4, 2, 1), (8, 4, 2, 16), (64, 12, 6, 1), (64, 12, 6, 8),
                                     (64, 12, 6, 64), (5, 2, 1, 3)])
def test_cache_decisions_bit_exact(E, B, K, T, policy):
    steps = 512 if T < 64 else 128
    ids = _stream_ids(E, K, T, steps, max(B // 2, K), seed=E + B + K + T)
    c = M.mcft_cache_create(1, E, B, max_assign=T * K, policy=policy)
    ref = oracle.cache.SlotCache(E, B, policy)
    d_ids = torch.from_numpy(ids).to(DEV)
    th = tf = tb = 0
    for s in range(steps):
        M.mcft_cache_step(c, 0, d_ids[s])
        M.mcft_fetch_experts(c, 0)
        h, f, b, ml = ref.step(ids[s])
        assert M.mcft_cache_last_misses(c, 0) == ml, f"step {s}"
        th, tf, tb = th + h, tf + f, tb + b
    assert M.mcft_cache_stats(c, 0) == (th, tf, tb)
    assert M.mcft_cache_tags(c, 0) == ref.tag
    M.mcft_device_error()


def test_cache_multi_layer_interleaved():
    L, E, B, K = 4, 8, 4, 2
    ids = [_stream_ids(E, K, 1, 300, 4, seed=100 + l) for l in range(L)]
    c = M.mcft_cache_create(L, E, B, max_assign=K)
    refs = [oracle.cache.LRUStamps(E, B) for _ in range(L)]
    tot = np.zeros(3, np.int64)
    for s in range(300):
        for l in range(L):
            M.mcft_cache_step(c, l, torch.from_numpy(ids[l][s]).to(DEV))
            M.mcft_fetch_experts(c, l)
            h, f, b, ml = refs[l].step(ids[l][s])
            assert M.mcft_cache_last_misses(c, l) == ml
            tot += (h, f, b)
    assert M.mcft_cache_stats(c, -1) == tuple(int(v) for v in tot)
    # batch 1: Fetches/tok = L K (1 - HR)  (Eq. metrics)
    hr, fpt = oracle.cache.metrics(tot[0], tot[1], 300, L, K)
    assert fpt == pytest.approx(L * K * (1 - hr))


def test_cache_fetch_copies_expert_bytes():
    """Misses copy the pinned host block of the expert into its slot (or a staging buffer for a
    bypass); the returned addresses hold exactly the selected experts' bytes."""
    L, E, B, K, T = 2, 8, 3, 2, 4
    nbytes = 3 * 64 * 64 * 2
    g = torch.Generator().manual_seed(0)
    host = [torch.randint(-2**31, 2**31 - 1, (nbytes // 4,), generator=g, dtype=torch.int32).pin_memory()
            for _ in range(L * E)]
    c = M.mcft_cache_create(L, E, B, nbytes, host, max_assign=T * K)
    ids = _stream_ids(E, K, T, 60, 4, seed=7)
    compute = torch.cuda.current_stream()
    copy = torch.cuda.Stream()
    for s in range(60):
        for l in range(L):
            M.mcft_cache_step(c, l, torch.from_numpy(ids[s]).to(DEV))
            ptrs = M.mcft_fetch_experts(c, l, compute, copy)
            used = set(ids[s].reshape(-1).tolist())
            for e in range(E):
                assert (ptrs[e] != 0) == (e in used)
            torch.cuda.synchronize()
            for e in used:
                buf = device_view(ptrs[e], nbytes // 4, torch.int32)
                assert torch.equal(buf.cpu(), host[l * E + e]), f"step {s} layer {l} expert {e}"
    M.mcft_device_error()


@pytest.mark.parametrize("nbytes,blocks", [(16, 1), (65536, 1), (65536 + 48, 3),
                                           (5 * 65536 + 16 * 77, 38), (17301504, 152)])
def test_host_copy_moves_every_byte(nbytes, blocks):
    """The link probe's SM-load copy: whole and ragged 64 KB pieces, grids smaller and larger than
    the piece count; the bytes after the copied range stay untouched."""
    g = torch.Generator().manual_seed(nbytes)
    src = torch.randint(0, 256, (nbytes,), generator=g, dtype=torch.uint8).pin_memory()
    dst = torch.full((nbytes + 64,), 0xAB, dtype=torch.uint8, device=DEV)
    M.mcft_host_copy(dst[:nbytes], src, blocks)
    torch.cuda.synchronize()
    assert torch.equal(dst[:nbytes].cpu(), src)
    assert bool((dst[nbytes:] == 0xAB).all())


@pytest.mark.parametrize("policy", ["LRU", "LFU", "FIFO"])
def test_cache_export_import_resume(policy):
    """Run N steps == run n steps, export, import into a fresh cache, run the other N - n."""
    E, B, K, T = 64, 12, 6, 8
    ids = _stream_ids(E, K, T, 200, 16, seed=9)
    d_ids = torch.from_numpy(ids).to(DEV)
    full = M.mcft_cache_create(1, E, B, max_assign=T * K, policy=policy)
    for s in range(200):
        M.mcft_cache_step(full, 0, d_ids[s])
    a = M.mcft_cache_create(1, E, B, max_assign=T * K, policy=policy)
    for s in range(77):
        M.mcft_cache_step(a, 0, d_ids[s])
    state = M.mcft_cache_export(a)
    b = M.mcft_cache_create(1, E, B, max_assign=T * K, policy=policy)
    M.mcft_cache_import(b, state)
    for s in range(77, 200):
        M.mcft_cache_step(b, 0, d_ids[s])
    assert M.mcft_cache_stats(b, 0) == M.mcft_cache_stats(full, 0)
    assert M.mcft_cache_tags(b, 0) == M.mcft_cache_tags(full, 0)
    other = M.mcft_cache_create(1, E, B + 1, max_assign=T * K, policy=policy)
    with pytest.raises(M.MCFTError):
        M.mcft_cache_import(other, state)
    other_policy = M.mcft_cache_create(1, E, B, max_assign=T * K,
                                       policy="FIFO" if policy != "FIFO" else "LRU")
    with pytest.raises(M.MCFTError):
        M.mcft_cache_import(other_policy, state)


def test_cache_bad_id_changes_nothing():
    c = M.mcft_cache_create(1, 8, 4, max_assign=4)
    M.mcft_cache_step(c, 0, torch.tensor([[1, 2]], dtype=torch.int32, device=DEV))
    M.mcft_fetch_experts(c, 0)
    before = (M.mcft_cache_stats(c, 0), M.mcft_cache_tags(c, 0))
    M.mcft_cache_step(c, 0, torch.tensor([[3, 9]], dtype=torch.int32, device=DEV))
    with pytest.raises(M.MCFTError) as ei:
        M.mcft_device_error()
    assert ei.value.status == M.MCFT_ERR_INVALID
    assert (M.mcft_cache_stats(c, 0), M.mcft_cache_tags(c, 0)) == before
    with pytest.raises(M.MCFTError):
        M.mcft_cache_step(c, 0, torch.zeros((3, 2), dtype=torch.int32, device=DEV))  # > max_assign
