"""Residual update and RMSNorm of the chained stack (mcft_residual_rmsnorm) against the oracle.

x <- x + y is one fp32 rounding of an exact sum, so it must match bit for bit. u = RMSNorm(x) is
compared with the fp64 oracle: fp32 within 1e-5 row-wise relative (a sum of d squares in fp32,
then one square root and three products); bf16 within one bf16 rounding (2^-8 relative, twice the
round-to-nearest bound) plus 1e-5 of the row's largest value for the fp32 part."""
import numpy as np
import pytest
import torch

import oracle
from paper_2609_34077_gb300 import inputs as I
from paper_2609_34077_gb300 import mcft as M
from tests.gpu_helpers import f64

pytestmark = pytest.mark.gpu
DEV = "cuda"
SHAPES = [I.TINY, I.MIXTRAL, I.DSV2_LITE]


def _inputs(shape, T):
    x = torch.from_numpy(I.normal_f32(1, ("norm-x", shape.name, T), T * shape.d, 3.0)
                         .reshape(T, shape.d))
    y = I.hidden_iid(2, shape, T, tag=("norm-y", T))
    gamma = I.norm_weight(3, shape, layer=T)
    return x, y, gamma


def _check_u(u_gpu, ref, dtype):
    got = f64(u_gpu)
    rowmax = np.abs(ref).max(axis=1, keepdims=True)
    if dtype == I.BF16:
        assert np.all(np.abs(got - ref) <= 2.0 ** -8 * np.abs(ref) + 1e-5 * rowmax)
    else:
        assert (np.abs(got - ref).max(axis=1) / rowmax[:, 0]).max() <= 1e-5


@pytest.mark.parametrize("T", [1, 7, 64])
@pytest.mark.parametrize("shape", SHAPES, ids=[s.name for s in SHAPES])
def test_residual_then_norm(shape, T):
    desc = M.desc_of(shape)
    x, y, gamma = _inputs(shape, T)
    xd, yd, gd = x.to(DEV), y.to(DEV), gamma.to(DEV)
    u = M.mcft_residual_rmsnorm(desc, xd, yd, gd, eps=shape.norm_eps)
    torch.cuda.synchronize()
    ref_x = (x.double() + y.double()).float()
    assert torch.equal(xd.cpu(), ref_x)
    _check_u(u, oracle.stack.rmsnorm(f64(ref_x), f64(gamma), shape.norm_eps), shape.dtype)


@pytest.mark.parametrize("shape", SHAPES, ids=[s.name for s in SHAPES])
def test_norm_only_and_add_only(shape):
    desc = M.desc_of(shape)
    T = 5
    x, y, gamma = _inputs(shape, T)
    xd = x.to(DEV)
    u = M.mcft_residual_rmsnorm(desc, xd, None, gamma.to(DEV), eps=shape.norm_eps)
    torch.cuda.synchronize()
    assert torch.equal(xd.cpu(), x)  # no y: the stream is untouched
    _check_u(u, oracle.stack.rmsnorm(f64(x), f64(gamma), shape.norm_eps), shape.dtype)
    out = M.mcft_residual_rmsnorm(desc, xd, y.to(DEV), None, eps=shape.norm_eps)
    torch.cuda.synchronize()
    assert out is None  # no gamma: only the residual update
    assert torch.equal(xd.cpu(), (x.double() + y.double()).float())


def test_zero_row_and_large_values():
    """A zero row normalises to zero (eps keeps it finite); rows of very different magnitude
    normalise to the same direction (scale invariance up to eps)."""
    shape = I.TINY
    desc = M.desc_of(shape)
    base = torch.from_numpy(I.normal_f32(4, "norm-scale", shape.d))
    x = torch.stack([torch.zeros(shape.d), base, base * 1e3, base * 1e-2])
    gamma = torch.ones(shape.d)
    u = M.mcft_residual_rmsnorm(desc, x.to(DEV), None, gamma.to(DEV), eps=1e-12)
    torch.cuda.synchronize()
    got = f64(u)
    assert np.all(got[0] == 0.0)
    for r in (2, 3):
        np.testing.assert_allclose(got[r], got[1], rtol=1e-5, atol=1e-6)


def test_invalid_arguments():
    desc = M.desc_of(I.TINY)
    x = torch.zeros((4, I.TINY.d), device=DEV)
    g = torch.ones(I.TINY.d, device=DEV)
    with pytest.raises(M.MCFTError):  # misaligned stream pointer
        M.mcft_residual_rmsnorm(desc, x.view(-1)[1:1 + 3 * I.TINY.d].view(3, I.TINY.d), None, g)
    with pytest.raises(M.MCFTError):
        M.mcft_residual_rmsnorm(desc, x, None, g, eps=-1.0)
