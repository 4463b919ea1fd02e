"""The C-ABI library builds, loads and exports every symbol include/mcft.h declares; host-side
argument checks that run before any CUDA call (no GPU needed)."""
import ctypes as C
import os
import re
import subprocess

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "mcft.h")


@pytest.fixture(scope="module")
def libpath():
    from paper_2609_34077_gb300 import build

    return build.build()


def declared():
    src = open(HEADER).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(mcft_\w+)\s*\(", src)))


def test_header_declares_the_four_paper_calls():
    names = declared()
    for n in ("mcft_route", "mcft_moe_forward", "mcft_cache_step", "mcft_fetch_experts"):
        assert n in names


def test_exports_match_header(libpath):
    out = subprocess.run(["nm", "-D", "--defined-only", libpath], capture_output=True, text=True,
                         check=True).stdout
    exported = set(re.findall(r"\bT (mcft_\w+)", out))
    assert set(declared()) <= exported
    lib = C.CDLL(libpath)
    for n in declared():
        getattr(lib, n)


def test_binding_covers_header(libpath):
    from paper_2609_34077_gb300 import mcft

    assert set(mcft.SIGNATURES) == set(declared())
    assert mcft.mcft_version() >= 100


def test_host_validation_without_gpu(libpath):
    from paper_2609_34077_gb300 import inputs, mcft

    L = mcft.lib()
    desc = mcft.desc_of(inputs.MIXTRAL)
    n = C.c_size_t(0)
    assert L.mcft_moe_workspace_size(C.byref(desc), 4096, C.byref(n)) == mcft.MCFT_OK
    assert n.value > 4096 * 2 * 14336 * 2  # holds the bf16 hidden activations
    bad = mcft.LayerDesc(4000, 8, 2, 14336, 0, 0, 1)  # d not a multiple of 64
    assert L.mcft_moe_workspace_size(C.byref(bad), 16, C.byref(n)) == mcft.MCFT_ERR_INVALID
    assert b"multiple of 64" in L.mcft_last_error()
    big = mcft.LayerDesc(4096, 128, 2, 14336, 0, 0, 1)
    assert L.mcft_moe_workspace_size(C.byref(big), 16, C.byref(n)) == mcft.MCFT_ERR_UNSUPPORTED
    # hard mask with fewer than K ones: rejected before any launch
    m = C.create_string_buffer(bytes([1, 0, 0, 0, 0, 0, 0, 0]), 8)
    st = L.mcft_route(C.byref(desc), C.c_void_p(16), 1, C.c_void_p(16), mcft.MCFT_ROUTE_HARD_MASK,
                      C.cast(m, C.c_void_p), None, C.c_void_p(16), C.c_void_p(16), None)
    assert st == mcft.MCFT_ERR_INVALID and b"fewer than K" in L.mcft_last_error()
    # a prior entry <= 0 is rejected (Eq. inference needs pi > 0)
    pr = (C.c_float * 8)(*([0.1] * 7 + [0.0]))
    st = L.mcft_route(C.byref(desc), C.c_void_p(16), 1, C.c_void_p(16), mcft.MCFT_ROUTE_SOFT_PRIOR,
                      None, C.cast(pr, C.c_void_p), C.c_void_p(16), C.c_void_p(16), None)
    assert st == mcft.MCFT_ERR_INVALID
    # cache: K <= B < E
    h = C.c_void_p()
    assert L.mcft_cache_create(1, 8, 8, 0, None, 2, 0, C.byref(h)) == mcft.MCFT_ERR_INVALID
    assert L.mcft_cache_create(1, 8, 0, 0, None, 2, 0, C.byref(h)) == mcft.MCFT_ERR_INVALID
    assert L.mcft_cache_create(1, 8, 4, 0, None, 2, 7, C.byref(h)) == mcft.MCFT_ERR_INVALID
    assert b"policy" in L.mcft_last_error()
    # host copy probe: alignment, size and grid are checked before any CUDA call
    assert L.mcft_host_copy(None, C.c_void_p(16), 16, 1, None) == mcft.MCFT_ERR_INVALID
    assert L.mcft_host_copy(C.c_void_p(16), C.c_void_p(24), 16, 1, None) == mcft.MCFT_ERR_INVALID
    assert b"aligned" in L.mcft_last_error()
    assert L.mcft_host_copy(C.c_void_p(16), C.c_void_p(32), 40, 1, None) == mcft.MCFT_ERR_INVALID
    assert b"multiple of 16" in L.mcft_last_error()
    assert L.mcft_host_copy(C.c_void_p(16), C.c_void_p(32), 64, 0, None) == mcft.MCFT_ERR_INVALID


def test_test_inject_validation_without_gpu(libpath):
    from paper_2609_34077_gb300 import mcft

    L = mcft.lib()
    assert L.mcft_test_inject(-1, 0, 0, 0) == mcft.MCFT_ERR_INVALID
    assert L.mcft_test_inject(0, -2, 0, 0) == mcft.MCFT_ERR_INVALID
    assert L.mcft_test_inject(0, 0, 0, 0) == mcft.MCFT_OK


def test_tc_tile_mode_without_gpu(libpath):
    """mcft_set_tc_tiles: only the two modes; under CTA-pair tiles a layer whose routed experts
    average >= 512 rows pads its segments to 256 rows (a larger workspace), a smaller one keeps
    the one-CTA layout, and a layer with adapters always does."""
    import ctypes as C
    from paper_2609_34077_gb300 import inputs as I
    from paper_2609_34077_gb300 import mcft

    L = mcft.lib()
    assert L.mcft_set_tc_tiles(2) == mcft.MCFT_ERR_INVALID
    assert L.mcft_set_tc_tiles(-1) == mcft.MCFT_ERR_INVALID
    desc = mcft.desc_of(I.MIXTRAL)

    def size(T):
        n = C.c_size_t(0)
        assert L.mcft_moe_workspace_size(C.byref(desc), T, C.byref(n)) == mcft.MCFT_OK
        return n.value

    def size_lora(T):
        n = C.c_size_t(0)
        assert L.mcft_moe_workspace_size_lora(C.byref(desc), 8, T, C.byref(n)) == mcft.MCFT_OK
        return n.value

    try:
        one = {T: size(T) for T in (1024, 2048, 4096)}
        one_lora = size_lora(4096)
        assert L.mcft_set_tc_tiles(mcft.MCFT_TC_TILES_CTA_PAIR) == mcft.MCFT_OK
        pair = {T: size(T) for T in (1024, 2048, 4096)}
        assert size_lora(4096) == one_lora
    finally:
        assert L.mcft_set_tc_tiles(mcft.MCFT_TC_TILES_ONE_CTA) == mcft.MCFT_OK
    assert pair[1024] == one[1024]  # 2048 assignments over 8 experts: 256 rows each
    assert pair[2048] > one[2048] and pair[4096] > one[4096]
    assert size(4096) == one[4096]


def test_read_probe_validation_without_gpu(libpath):
    import ctypes as C
    from paper_2609_34077_gb300 import mcft

    L = mcft.lib()
    buf, sink = C.c_void_p(4096), C.c_void_p(64)
    assert L.mcft_read_probe(None, 16, 0, 0, 1, sink, None) == mcft.MCFT_ERR_INVALID
    assert L.mcft_read_probe(buf, 16, 0, 0, 1, None, None) == mcft.MCFT_ERR_INVALID
    assert L.mcft_read_probe(C.c_void_p(4100), 16, 0, 0, 1, sink, None) == mcft.MCFT_ERR_INVALID
    assert L.mcft_read_probe(buf, 16, 2, 0, 1, sink, None) == mcft.MCFT_ERR_INVALID
    assert L.mcft_read_probe(buf, 24, 0, 0, 1, sink, None) == mcft.MCFT_ERR_INVALID
    assert L.mcft_read_probe(buf, 32 * 4096, 1, 100, 1, sink, None) == mcft.MCFT_ERR_INVALID
    assert L.mcft_read_probe(buf, 32 * 4096 + 16, 1, 4096, 1, sink, None) == mcft.MCFT_ERR_INVALID
    assert L.mcft_read_probe(buf, 16, 0, 0, 0, sink, None) == mcft.MCFT_ERR_INVALID
    assert L.mcft_read_probe(buf, 0, 0, 0, 1, sink, None) == mcft.MCFT_OK  # nothing to read
