"""The HBM read probe (mcft_read_probe) reads every 32-bit word of its buffer exactly once, in
both of its patterns: the XOR it folds into its sink equals the buffer's XOR computed on the host.
(A word read twice would cancel out of the XOR, a word skipped would be missing from it.)"""
import numpy as np
import pytest
import torch

from paper_2609_34077_gb300 import mcft as M

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("pattern,row_bytes,nbytes", [(0, 4096, 4 << 20), (0, 4096, (4 << 20) + 48),
                                                      (1, 4096, 32 * 4096 * 37),
                                                      (1, 8192, 32 * 8192 * 5),
                                                      (1, 2816, 32 * 2816 * 3)])
def test_read_probe_reads_every_word_once(pattern, row_bytes, nbytes):
    rng = np.random.default_rng(pattern * 1000 + row_bytes)
    host = rng.integers(0, 2 ** 32, size=nbytes // 4, dtype=np.uint64).astype(np.uint32)
    expect = np.bitwise_xor.reduce(host)
    buf = torch.from_numpy(host.view(np.int32)).to("cuda")
    for blocks in (1, 7, 304):
        sink = M.mcft_read_probe(buf, pattern, row_bytes=row_bytes, blocks=blocks)
        M.mcft_device_error()
        got = np.uint32(sink.cpu().numpy().view(np.uint32)[0])
        assert got == expect, f"pattern {pattern} blocks {blocks}"
