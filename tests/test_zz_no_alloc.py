"""mcft_moe_forward_noalloc against mcft_moe_forward, through the C ABI.

Some callers cannot allocate device memory when they run a layer: a plugin inside an application
that owns every device allocation through its own pool, or a decode loop that cannot take an
allocation's implicit synchronisation. mcft_moe_forward_noalloc serves them from a fixed scratch
array inside the library instead of a caller-provided workspace. These tests check that two calls
in a row (the array keeps the previous call's contents) give exactly the bits of the workspace
entry point (both run the same kernels with the same workspace layout, so any difference, even in
the low bits, would mean stale scratch leaking into a call), and that a call needing more scratch
than the array holds is refused. This file is collected last on purpose.
"""
import numpy as np
import pytest
import torch

from paper_2609_34077_gb300 import inputs as I
from paper_2609_34077_gb300 import mcft as M
from tests.gpu_helpers import TOL_BF16, check_output, f64

pytestmark = pytest.mark.gpu
DEV = "cuda"

SMALL_MIX = I.LayerShape("noalloc-mix", d=512, E=8, K=2, w=384, n_shared=0, gate=I.GATE_RENORM,
                         dtype=I.BF16, cache_slots=4, keep=4)
SMALL_DS = I.LayerShape("noalloc-ds", d=256, E=64, K=6, w=128, n_shared=2, gate=I.GATE_PLAIN,
                        dtype=I.BF16, cache_slots=12, keep=16)


@pytest.mark.parametrize("shape,T", [(SMALL_MIX, 16), (SMALL_DS, 64), (I.MIXTRAL, 16)],
                         ids=["mix-small-T16", "ds-small-T64", "mixtral-T16"])
def test_noalloc_matches_workspace_forward_two_calls(shape, T):
    lw = I.layer_weights(40, shape)
    desc = M.desc_of(shape)
    experts = [b.to(DEV) for b in lw.experts]
    shared = [b.to(DEV) for b in lw.shared]
    for call in range(2):
        x = I.hidden_iid(41 + call, shape, T).to(DEV)
        ids = I.random_ids(42 + call, 1, T, shape.K, shape.E, hot=range(shape.keep))[0]
        idx = torch.from_numpy(ids).to(DEV)
        gate = torch.from_numpy(
            np.random.default_rng(43 + call).uniform(0.05, 1.0, (T, shape.K)).astype(np.float32)).to(DEV)
        y_ref = M.mcft_moe_forward(desc, x, idx, gate, experts, shared)
        y = M.mcft_moe_forward_noalloc(desc, x, idx, gate, experts, shared)
        M.mcft_device_error()
        assert torch.equal(y, y_ref), f"{shape.name} call {call}: outputs differ from the workspace call"
        check_output(y, f64(y_ref), TOL_BF16, f"{shape.name} call {call}")


def test_noalloc_refuses_calls_beyond_its_scratch():
    desc = M.desc_of(I.MIXTRAL)
    T = 4096  # prefill-sized: needs about 490 MB of scratch
    x = torch.zeros((T, I.MIXTRAL.d), dtype=torch.bfloat16, device=DEV)
    idx = torch.zeros((T, 2), dtype=torch.int32, device=DEV)
    gate = torch.zeros((T, 2), dtype=torch.float32, device=DEV)
    with pytest.raises(M.MCFTError) as ei:
        M.mcft_moe_forward_noalloc(desc, x, idx, gate, [None] * 8)
    assert ei.value.status == M.MCFT_ERR_UNSUPPORTED
    assert "scratch" in str(ei.value)
    M.mcft_device_error()
