"""Failure paths, made to happen on the host or by a bounded wait that runs out (never by a GPU
fault): a pinned host allocation the runtime refuses (mcft_cache_create returns MCFT_ERR_OOM and
frees what it had allocated), an expert copy the runtime refuses (mcft_fetch_experts returns
MCFT_ERR_CUDA and the cache can still be destroyed cleanly), and the fused decode FFN's wait for a
segment's GEMM13 items running out (MCFT_ERR_TIMEOUT through the device error word, the output left
untouched, the next call correct). Injection goes through mcft_test_inject and is switched off
again by every test, pass or fail."""
import numpy as np
import pytest
import torch

import oracle
from paper_2609_34077_gb300 import inputs as I
from paper_2609_34077_gb300 import mcft as M
from tests.gpu_helpers import TOL_BF16, check_output, expert_triples, f64, shared_triples

pytestmark = pytest.mark.gpu
DEV = "cuda"

SMALL_DS = I.LayerShape("faults-ds", d=256, E=64, K=6, w=128, n_shared=2, gate=I.GATE_PLAIN,
                        dtype=I.BF16, cache_slots=12, keep=16)


@pytest.fixture(autouse=True)
def _injection_off():
    M.mcft_test_inject()
    yield
    M.mcft_test_inject()


def test_pinned_allocation_failure_returns_oom():
    M.mcft_test_inject(fail_pinned_allocs=1)
    with pytest.raises(M.MCFTError) as ei:
        M.mcft_cache_create(2, 8, 4, max_assign=2)
    assert ei.value.status == M.MCFT_ERR_OOM
    M.mcft_test_inject()
    c = M.mcft_cache_create(2, 8, 4, max_assign=2)  # nothing leaked or left half-built
    M.mcft_cache_step(c, 0, torch.tensor([[1, 2]], dtype=torch.int32, device=DEV))
    M.mcft_fetch_experts(c, 0)
    assert M.mcft_cache_stats(c, 0) == (0, 2, 0)
    M.mcft_cache_destroy(c)
    M.mcft_device_error()


def test_expert_copy_failure_returns_cuda_error_and_destroys_cleanly():
    L, E, B, K = 1, 8, 3, 2
    nbytes = 3 * 64 * 64 * 2
    host = [torch.full((nbytes // 2,), e, dtype=torch.int16).pin_memory() for e in range(E)]
    c = M.mcft_cache_create(L, E, B, nbytes, host, max_assign=K)
    compute, copy = torch.cuda.current_stream(), torch.cuda.Stream()
    M.mcft_cache_step(c, 0, torch.tensor([[3, 5]], dtype=torch.int32, device=DEV))
    M.mcft_test_inject(fail_expert_copies=1)
    with pytest.raises(M.MCFTError) as ei:
        M.mcft_fetch_experts(c, 0, compute, copy)
    assert ei.value.status == M.MCFT_ERR_CUDA
    M.mcft_test_inject()
    M.mcft_cache_destroy(c)
    M.mcft_device_error()
    # a fresh cache works, and its fetches land
    c = M.mcft_cache_create(L, E, B, nbytes, host, max_assign=K)
    M.mcft_cache_step(c, 0, torch.tensor([[3, 5]], dtype=torch.int32, device=DEV))
    ptrs = M.mcft_fetch_experts(c, 0, compute, copy)
    torch.cuda.synchronize()
    from tests.gpu_helpers import device_view

    for e in (3, 5):
        got = device_view(ptrs[e], nbytes // 4, torch.int32).cpu()
        assert torch.equal(got, host[e].view(torch.int32))
    M.mcft_cache_destroy(c)
    M.mcft_device_error()


@pytest.mark.parametrize("T", [1, 16, 64])
def test_decode_ffn_wait_runs_out(T):
    """With its GEMM13 items withheld, every GEMM2 item of the fused decode FFN waits for a segment
    that never completes; the 1 ms limit ends the wait, the call reports MCFT_ERR_TIMEOUT and y is
    untouched; with injection off the same call on the same workspace is correct."""
    sh = SMALL_DS
    lw = I.layer_weights(95, sh)
    desc = M.desc_of(sh)
    x = I.hidden_iid(95, sh, T)
    ids = I.random_ids(95, 1, T, sh.K, sh.E, hot=range(sh.keep))[0]
    idx = torch.from_numpy(ids).to(DEV)
    gate = torch.from_numpy(np.random.default_rng(95).uniform(0.05, 1.0, (T, sh.K))
                            .astype(np.float32)).to(DEV)
    experts = [b.to(DEV) for b in lw.experts]
    shared = [b.to(DEV) for b in lw.shared]
    ws = torch.empty(M.mcft_moe_workspace_size(desc, T), dtype=torch.uint8, device=DEV)
    y = torch.full((T, sh.d), 7.0, dtype=torch.bfloat16, device=DEV)
    M.mcft_test_inject(wait_limit_ns=1_000_000, withhold_gemm13=True)
    M.mcft_moe_forward(desc, x.to(DEV), idx, gate, experts, shared, y=y, workspace=ws)
    M.mcft_test_inject()
    with pytest.raises(M.MCFTError) as ei:
        M.mcft_device_error()
    assert ei.value.status == M.MCFT_ERR_TIMEOUT
    assert torch.all(y == 7.0)
    M.mcft_moe_forward(desc, x.to(DEV), idx, gate, experts, shared, y=y, workspace=ws)
    M.mcft_device_error()
    ref = oracle.ffn.moe_layer(f64(x), ids, gate.cpu().double().numpy(), expert_triples(lw, sh),
                               shared_triples(lw, sh))
    check_output(y, ref, TOL_BF16, f"after the timeout, T={T}")


def test_cached_forward_wait_runs_out_and_the_cache_stays_whole():
    """The cached forward at batch 1 fetches its misses in the FFN's own launch. With GEMM13 items
    withheld and a 1 ms wait limit, that launch's GEMM2 waits run out: MCFT_ERR_TIMEOUT, y untouched.
    Its fetchers still copy every missed block (the cache already counts them as resident), so the
    following steps, with injection off, equal the plain forward bit for bit."""
    sh = SMALL_DS
    lw = I.layer_weights(96, sh, pin=True)
    desc = M.desc_of(sh)
    cache = M.mcft_cache_create(1, sh.E, sh.cache_slots, sh.expert_bytes, lw.experts, max_assign=sh.K)
    experts = [b.to(DEV) for b in lw.experts]
    shared = [b.to(DEV) for b in lw.shared]
    ws = torch.empty(M.mcft_moe_workspace_size(desc, 1), dtype=torch.uint8, device=DEV)
    compute, copy = torch.cuda.Stream(), torch.cuda.Stream()
    ids = I.random_ids(96, 6, 1, sh.K, sh.E, hot=range(sh.keep), p_hot=0.7)
    for s in range(6):
        x = I.hidden_iid(97 + s, sh, 1).to(DEV)
        idx = torch.from_numpy(ids[s]).to(DEV)
        gate = torch.full((1, sh.K), 0.25, device=DEV)
        y = torch.full((1, sh.d), 7.0, dtype=torch.bfloat16, device=DEV)
        torch.cuda.synchronize()
        M.mcft_cache_step(cache, 0, idx, stream=compute)
        if s == 0:
            M.mcft_test_inject(wait_limit_ns=1_000_000, withhold_gemm13=True)
        M.mcft_moe_forward_cached(desc, x, idx, gate, cache, 0, shared, y=y, workspace=ws,
                                  compute_stream=compute, copy_stream=copy)
        M.mcft_test_inject()
        compute.synchronize()
        if s == 0:
            with pytest.raises(M.MCFTError) as ei:
                M.mcft_device_error()
            assert ei.value.status == M.MCFT_ERR_TIMEOUT
            assert torch.all(y == 7.0)
            continue
        M.mcft_device_error()
        y_ref = M.mcft_moe_forward(desc, x, idx, gate, experts, shared)
        assert torch.equal(y, y_ref), f"step {s}"
    assert M.mcft_cache_stats(cache, 0)[1] > sh.K  # the stream kept fetching
