"""Python binding of libmcft (C ABI in include/mcft.h): argument marshalling only.

Every function here has the name of the C entry point it calls and does nothing but convert torch
tensors and Python values into pointers and sizes. All computation runs in libmcft.so; if the
library is missing this module raises instead of computing anything another way.
"""
from __future__ import annotations

import ctypes as C
import os

import torch

_LIB_PATH = os.path.join(os.path.dirname(os.path.abspath(__file__)), "libmcft.so")

MCFT_OK, MCFT_ERR_INVALID, MCFT_ERR_OOM, MCFT_ERR_CUDA, MCFT_ERR_TIMEOUT, MCFT_ERR_UNSUPPORTED = range(6)
MCFT_ROUTE_TOPK, MCFT_ROUTE_HARD_MASK, MCFT_ROUTE_SOFT_PRIOR = 0, 1, 2
MCFT_GATE_RENORM, MCFT_GATE_PLAIN = 0, 1
MCFT_F32, MCFT_BF16 = 0, 1
MCFT_CACHE_LRU, MCFT_CACHE_LFU, MCFT_CACHE_FIFO = 0, 1, 2
POLICY = {"LRU": MCFT_CACHE_LRU, "LFU": MCFT_CACHE_LFU, "FIFO": MCFT_CACHE_FIFO}

# every exported entry point: name -> (restype, argtypes)
_vp, _i, _sz = C.c_void_p, C.c_int, C.c_size_t
SIGNATURES = {
    "mcft_route": (_i, [_vp, _vp, _i, _vp, _i, _vp, _vp, _vp, _vp, _vp]),
    "mcft_moe_workspace_size": (_i, [_vp, _i, C.POINTER(_sz)]),
    "mcft_moe_forward": (_i, [_vp, _vp, _i, _vp, _vp, _vp, _vp, _vp, _vp, _sz, _vp]),
    "mcft_moe_forward_noalloc": (_i, [_vp, _vp, _i, _vp, _vp, _vp, _vp, _vp, _vp]),
    "mcft_moe_workspace_size_lora": (_i, [_vp, _i, _i, C.POINTER(_sz)]),
    "mcft_moe_forward_lora": (_i, [_vp, _vp, _i, _vp, _vp, _vp, _vp, _vp, _vp, _i, C.c_float, _vp, _vp,
                                   _sz, _vp]),
    "mcft_cache_create": (_i, [_i, _i, _i, _sz, _vp, _i, _i, C.POINTER(_vp)]),
    "mcft_cache_step": (_i, [_vp, _i, _vp, _i, _i, _vp]),
    "mcft_fetch_experts": (_i, [_vp, _i, _vp, _vp, _vp]),
    "mcft_host_copy": (_i, [_vp, _vp, _sz, _i, _vp]),
    "mcft_moe_forward_cached": (_i, [_vp, _vp, _i, _vp, _vp, _vp, _i, _vp, _vp, _vp, _sz, _vp, _vp]),
    "mcft_mask_sample": (_i, [_vp, _vp, _i, _i, _i, _vp, _vp, _vp]),
    "mcft_gate_grad": (_i, [_vp, _vp, _i, _vp, _sz, _vp, _vp]),
    "mcft_mask_grad": (_i, [_vp, _vp, _vp, _vp, _i, _vp, _vp, _vp, _i, _vp]),
    "mcft_cache_last_misses": (_i, [_vp, _i, C.POINTER(_i), _vp, _vp]),
    "mcft_cache_stats": (_i, [_vp, _i, C.POINTER(C.c_uint64), C.POINTER(C.c_uint64),
                              C.POINTER(C.c_uint64), _vp]),
    "mcft_cache_tags": (_i, [_vp, _i, _vp, _vp]),
    "mcft_cache_prefetch": (_i, [_vp, _i, _vp, _i, _i, _i, _vp]),
    "mcft_cache_prefetch_stats": (_i, [_vp, _i, C.POINTER(C.c_uint64), C.POINTER(C.c_uint64),
                                       C.POINTER(C.c_uint64), _vp]),
    "mcft_residual_rmsnorm": (_i, [_vp, _vp, _vp, _i, _vp, C.c_float, _vp, _vp]),
    "mcft_stack_create": (_i, [_vp, _i, _vp, _vp, _vp, _vp, C.c_float, _vp, _i, _i, C.POINTER(_vp)]),
    "mcft_stack_step": (_i, [_vp, _vp, _i, _vp, _vp]),
    "mcft_stack_routing": (_i, [_vp, _i, _vp, _vp, _vp, _vp]),
    "mcft_stack_destroy": (None, [_vp]),
    "mcft_cache_export": (_i, [_vp, _vp, C.POINTER(_sz), _vp]),
    "mcft_cache_import": (_i, [_vp, _vp, _sz, _vp]),
    "mcft_cache_destroy": (None, [_vp]),
    "mcft_device_error": (_i, [_vp]),
    "mcft_test_inject": (_i, [_i, _i, C.c_ulonglong, _i]),
    "mcft_profile_enable": (_i, [_i]),
    "mcft_set_tc_tiles": (_i, [_i]),
    "mcft_read_probe": (_i, [_vp, _sz, _i, _i, _i, _vp, _vp]),
    "mcft_profile_reset": (_i, []),
    "mcft_profile_read": (_i, [_i, _vp, _vp, _vp, C.POINTER(_i)]),
    "mcft_last_error": (C.c_char_p, []),
    "mcft_version": (_i, []),
}


class MCFTError(RuntimeError):
    def __init__(self, status, msg):
        super().__init__(f"mcft status {status}: {msg}")
        self.status = status


class LayerDesc(C.Structure):
    """mcft_layer_desc"""
    _fields_ = [("d", C.c_int), ("E", C.c_int), ("K", C.c_int), ("w", C.c_int),
                ("n_shared", C.c_int), ("gate", C.c_int), ("dtype", C.c_int)]


_lib = None


def lib():
    """Load libmcft.so (built by paper_2609_34077_gb300.build); raise if it is not there."""
    global _lib
    if _lib is None:
        if not os.path.exists(_LIB_PATH):
            raise RuntimeError(f"{_LIB_PATH} is missing: build it with "
                               "`python -c 'import __graft_entry__ as g; g.build()'`")
        L = C.CDLL(_LIB_PATH)
        for name, (res, args) in SIGNATURES.items():
            f = getattr(L, name)
            f.restype = res
            f.argtypes = args
        _lib = L
    return _lib


def _check(st):
    if st != MCFT_OK:
        raise MCFTError(st, lib().mcft_last_error().decode())


def _stream(stream):
    if stream is None:
        return C.c_void_p(torch.cuda.current_stream().cuda_stream)
    if isinstance(stream, torch.cuda.Stream):
        return C.c_void_p(stream.cuda_stream)
    return C.c_void_p(int(stream))


def _ptr(t):
    if t is None:
        return None
    if isinstance(t, int):
        return C.c_void_p(t)
    assert t.is_contiguous(), "tensors passed to libmcft must be contiguous"
    return C.c_void_p(t.data_ptr())


def desc_of(shape) -> LayerDesc:
    """mcft_layer_desc of an inputs.LayerShape."""
    return LayerDesc(shape.d, shape.E, shape.K, shape.w, shape.n_shared, shape.gate, shape.dtype)


def torch_dtype(desc: LayerDesc):
    return torch.bfloat16 if desc.dtype == MCFT_BF16 else torch.float32


def mcft_version() -> int:
    return lib().mcft_version()


def mcft_device_error(stream=None):
    _check(lib().mcft_device_error(_stream(stream)))


def mcft_route(desc: LayerDesc, x, w_router, mode, mask=None, prior=None, idx=None, gate=None,
               stream=None):
    """idx [T,K] int32 and gate [T,K] fp32 (allocated on x's device if not given)."""
    T = x.shape[0]
    if idx is None:
        idx = torch.empty((T, desc.K), dtype=torch.int32, device=x.device)
    if gate is None:
        gate = torch.empty((T, desc.K), dtype=torch.float32, device=x.device)
    m = None
    if mask is not None:
        mb = bytes(int(v) for v in mask)
        m = C.create_string_buffer(mb, len(mb))
    p = None
    if prior is not None:
        p = (C.c_float * desc.E)(*[float(v) for v in prior])
    _check(lib().mcft_route(C.byref(desc), _ptr(x), T, _ptr(w_router), int(mode),
                            C.cast(m, C.c_void_p) if m is not None else None,
                            C.cast(p, C.c_void_p) if p is not None else None,
                            _ptr(idx), _ptr(gate), _stream(stream)))
    return idx, gate


def mcft_moe_workspace_size(desc: LayerDesc, T_max: int) -> int:
    n = C.c_size_t(0)
    _check(lib().mcft_moe_workspace_size(C.byref(desc), int(T_max), C.byref(n)))
    return n.value


def _ptr_array(items, n):
    arr = (C.c_void_p * max(n, 1))()
    for i in range(n):
        it = items[i] if items is not None and i < len(items) else None
        arr[i] = None if it is None else (it if isinstance(it, int) else it.data_ptr())
    return arr


def mcft_moe_forward(desc: LayerDesc, x, idx, gate, experts, shared=(), y=None, workspace=None,
                     stream=None):
    """y [T,d] = sum_k gate F_idx(x) + shared experts. ``experts``: E tensors / device addresses /
    None; ``workspace``: uint8 device tensor (allocated if not given)."""
    T = x.shape[0]
    if y is None:
        y = torch.empty_like(x)
    if workspace is None:
        workspace = torch.empty(mcft_moe_workspace_size(desc, T), dtype=torch.uint8, device=x.device)
    ex = _ptr_array(experts, desc.E)
    sh = _ptr_array(shared, desc.n_shared)
    _check(lib().mcft_moe_forward(C.byref(desc), _ptr(x), T, _ptr(idx), _ptr(gate),
                                  C.cast(ex, C.c_void_p), C.cast(sh, C.c_void_p), _ptr(y),
                                  _ptr(workspace), workspace.numel(), _stream(stream)))
    return y


def mcft_moe_workspace_size_lora(desc: LayerDesc, rank: int, T_max: int) -> int:
    n = C.c_size_t(0)
    _check(lib().mcft_moe_workspace_size_lora(C.byref(desc), int(rank), int(T_max), C.byref(n)))
    return n.value


def mcft_moe_forward_lora(desc: LayerDesc, x, idx, gate, experts, shared=(), expert_lora=None,
                          shared_lora=None, rank=8, scale=2.0, y=None, workspace=None, stream=None):
    """Layer forward with LoRA adapters (packed blocks, see include/mcft.h) on the experts."""
    T = x.shape[0]
    if y is None:
        y = torch.empty_like(x)
    if workspace is None:
        workspace = torch.empty(mcft_moe_workspace_size_lora(desc, rank, T), dtype=torch.uint8,
                                device=x.device)
    ex = _ptr_array(experts, desc.E)
    sh = _ptr_array(shared, desc.n_shared)
    el = _ptr_array(expert_lora, desc.E)
    sl = _ptr_array(shared_lora, desc.n_shared)
    _check(lib().mcft_moe_forward_lora(C.byref(desc), _ptr(x), T, _ptr(idx), _ptr(gate),
                                       C.cast(ex, C.c_void_p), C.cast(sh, C.c_void_p),
                                       C.cast(el, C.c_void_p), C.cast(sl, C.c_void_p), int(rank),
                                       float(scale), _ptr(y), _ptr(workspace), workspace.numel(),
                                       _stream(stream)))
    return y


def mcft_moe_forward_noalloc(desc: LayerDesc, x, idx, gate, experts, shared=(), y=None, stream=None):
    """mcft_moe_forward without a workspace: the library's static scratch array is used instead
    (for callers that cannot allocate device memory; decode-sized calls only)."""
    T = x.shape[0]
    if y is None:
        y = torch.empty_like(x)
    ex = _ptr_array(experts, desc.E)
    sh = _ptr_array(shared, desc.n_shared)
    _check(lib().mcft_moe_forward_noalloc(C.byref(desc), _ptr(x), T, _ptr(idx), _ptr(gate),
                                          C.cast(ex, C.c_void_p), C.cast(sh, C.c_void_p), _ptr(y),
                                          _stream(stream)))
    return y


class Cache:
    """Handle of an mcft_cache (per-layer expert cache, Section 4.1)."""

    def __init__(self, handle, L, E, B):
        self.handle, self.L, self.E, self.B = handle, L, E, B

    def __del__(self):
        if getattr(self, "handle", None):
            try:
                mcft_cache_destroy(self)
            except Exception:
                pass


def mcft_cache_create(L, E, B, expert_bytes=0, host_experts=None, max_assign=1024,
                      policy=MCFT_CACHE_LRU) -> Cache:
    """host_experts: L*E pinned host tensors (layer-major) or None for accounting only;
    policy: MCFT_CACHE_LRU / LFU / FIFO or the names "LRU" / "LFU" / "FIFO"."""
    h = C.c_void_p()
    arr = _ptr_array(host_experts, L * E) if host_experts is not None else None
    pol = POLICY.get(policy, policy)
    _check(lib().mcft_cache_create(L, E, B, expert_bytes,
                                   C.cast(arr, C.c_void_p) if arr is not None else None,
                                   max_assign, int(pol), C.byref(h)))
    c = Cache(h.value, L, E, B)
    c._host_experts = host_experts  # keep the pinned blocks alive
    return c


def mcft_cache_destroy(cache: Cache):
    if cache.handle:
        lib().mcft_cache_destroy(C.c_void_p(cache.handle))
        cache.handle = None


def mcft_cache_step(cache: Cache, layer, idx, stream=None):
    T, K = idx.shape
    _check(lib().mcft_cache_step(C.c_void_p(cache.handle), layer, _ptr(idx), T, K, _stream(stream)))


def mcft_fetch_experts(cache: Cache, layer, compute_stream=None, copy_stream=None):
    """Returns the E device addresses (0 for experts not selected this step)."""
    out = (C.c_void_p * cache.E)()
    _check(lib().mcft_fetch_experts(C.c_void_p(cache.handle), layer, _stream(compute_stream),
                                    _stream(copy_stream), C.cast(out, C.c_void_p)))
    return [v or 0 for v in out]


def mcft_host_copy(dst, host_src, blocks, stream=None):
    """Copy the pinned host tensor host_src into the device tensor dst (same byte size) with the
    fetch kernel's copy loop on `blocks` CTAs."""
    nbytes = host_src.numel() * host_src.element_size()
    assert dst.numel() * dst.element_size() == nbytes, "dst and host_src differ in size"
    _check(lib().mcft_host_copy(_ptr(dst), _ptr(host_src), nbytes, int(blocks), _stream(stream)))
    return dst


def mcft_read_probe(buf, pattern, row_bytes=4096, blocks=None, sink=None, stream=None):
    """Read the device tensor buf in one launch (pattern 0: contiguous; 1: the decode FFN's weight
    loads over rows of row_bytes) with no computation; returns sink (an int32 device tensor of one
    element, XORed with the XOR of every 32-bit word read)."""
    nbytes = buf.numel() * buf.element_size()
    if blocks is None:
        blocks = 2 * torch.cuda.get_device_properties(buf.device).multi_processor_count
    if sink is None:
        sink = torch.zeros(1, dtype=torch.int32, device=buf.device)
    _check(lib().mcft_read_probe(_ptr(buf), nbytes, int(pattern), int(row_bytes), int(blocks),
                                 _ptr(sink), _stream(stream)))
    return sink


def mcft_moe_forward_cached(desc: LayerDesc, x, idx, gate, cache: Cache, layer, shared=(), y=None,
                            workspace=None, compute_stream=None, copy_stream=None):
    """Decode forward of `layer` with experts from the cache, fetch driven on the device."""
    T = x.shape[0]
    if y is None:
        y = torch.empty_like(x)
    if workspace is None:
        workspace = torch.empty(mcft_moe_workspace_size(desc, T), dtype=torch.uint8, device=x.device)
    sh = _ptr_array(shared, desc.n_shared)
    _check(lib().mcft_moe_forward_cached(C.byref(desc), _ptr(x), T, _ptr(idx), _ptr(gate),
                                         C.c_void_p(cache.handle), layer, C.cast(sh, C.c_void_p),
                                         _ptr(y), _ptr(workspace), workspace.numel(),
                                         _stream(compute_stream), _stream(copy_stream)))
    return y


def mcft_cache_last_misses(cache: Cache, layer):
    n = C.c_int(0)
    ex = (C.c_int32 * cache.E)()
    sl = (C.c_int32 * cache.E)()
    _check(lib().mcft_cache_last_misses(C.c_void_p(cache.handle), layer, C.byref(n),
                                        C.cast(ex, C.c_void_p), C.cast(sl, C.c_void_p)))
    return [(ex[i], sl[i]) for i in range(n.value)]


def mcft_cache_stats(cache: Cache, layer=-1, stream=None):
    h, f, b = C.c_uint64(), C.c_uint64(), C.c_uint64()
    _check(lib().mcft_cache_stats(C.c_void_p(cache.handle), layer, C.byref(h), C.byref(f),
                                  C.byref(b), _stream(stream)))
    return h.value, f.value, b.value


def mcft_cache_prefetch(cache: Cache, layer, idx_pred, n_max, stream=None):
    """Prefetch event of `layer` from the predicted routing idx_pred [T, K] int32 (device)."""
    T, K = idx_pred.shape
    _check(lib().mcft_cache_prefetch(C.c_void_p(cache.handle), layer, _ptr(idx_pred), T, K,
                                     int(n_max), _stream(stream)))


def mcft_cache_prefetch_stats(cache: Cache, layer=-1, stream=None):
    """(prefetched, useful, bytes_moved) cumulative for one layer or all layers (layer = -1)."""
    p, u, b = C.c_uint64(), C.c_uint64(), C.c_uint64()
    _check(lib().mcft_cache_prefetch_stats(C.c_void_p(cache.handle), layer, C.byref(p), C.byref(u),
                                           C.byref(b), _stream(stream)))
    return p.value, u.value, b.value


def mcft_residual_rmsnorm(desc: LayerDesc, x, y=None, gamma=None, eps=1e-5, u=None, stream=None):
    """x [T, d] fp32 (updated in place when y is given); returns u [T, d] in the layer dtype
    (allocated on x's device if not given) when gamma is given, else None."""
    T = x.shape[0]
    if gamma is not None and u is None:
        u = torch.empty((T, desc.d), dtype=torch.bfloat16 if desc.dtype == MCFT_BF16 else torch.float32,
                        device=x.device)
    _check(lib().mcft_residual_rmsnorm(C.byref(desc), _ptr(x), _ptr(y) if y is not None else None, T,
                                       _ptr(gamma) if gamma is not None else None, C.c_float(eps),
                                       _ptr(u) if gamma is not None else None, _stream(stream)))
    return u


class Stack:
    """Handle of an mcft_stack (chained decode stack over a cache)."""

    def __init__(self, handle, L, K, keep):
        self.handle, self.L, self.K, self._keep = handle, L, K, keep
        self.last_T = 0

    def __del__(self):
        if getattr(self, "handle", None):
            try:
                mcft_stack_destroy(self)
            except Exception:
                pass


def mcft_stack_create(desc: LayerDesc, routers, priors, gammas, shared, eps, cache: Cache,
                      n_prefetch=0, T_max=1) -> Stack:
    """routers, gammas: L device tensors; priors: [L, E] array-like (fp32 > 0); shared: L lists of
    S device blocks (or None when S = 0)."""
    L = len(routers)
    import numpy as _np
    pri = _np.ascontiguousarray(_np.asarray(priors, _np.float32).reshape(-1))
    rp = _ptr_array(routers, L)
    gp = _ptr_array(gammas, L)
    flat = [b for row in shared for b in row] if shared else []
    sp = _ptr_array(flat, len(flat))
    h = C.c_void_p()
    _check(lib().mcft_stack_create(C.byref(desc), L, C.cast(rp, C.c_void_p), pri.ctypes.data,
                                   C.cast(gp, C.c_void_p), C.cast(sp, C.c_void_p) if flat else None,
                                   C.c_float(eps), C.c_void_p(cache.handle), int(n_prefetch),
                                   int(T_max), C.byref(h)))
    # keep everything the stack points to alive with it
    return Stack(h.value, L, desc.K, (list(routers), list(gammas), flat, cache))


def mcft_stack_step(stack: Stack, x, compute_stream=None, copy_stream=None):
    """x [T, d] fp32 device tensor, updated in place (x_0 in, x_L out)."""
    T = x.shape[0]
    _check(lib().mcft_stack_step(C.c_void_p(stack.handle), _ptr(x), T, _stream(compute_stream),
                                 _stream(copy_stream)))
    stack.last_T = T


def mcft_stack_routing(stack: Stack, layer, stream=None):
    """(idx [T, K] int32, gate [T, K] fp32, idx_pred [T, K] int32) numpy copies of the last step."""
    import numpy as _np
    T, K = stack.last_T, stack.K
    idx = _np.empty((T, K), _np.int32)
    gate = _np.empty((T, K), _np.float32)
    pred = _np.empty((T, K), _np.int32)
    _check(lib().mcft_stack_routing(C.c_void_p(stack.handle), layer, idx.ctypes.data,
                                    gate.ctypes.data, pred.ctypes.data, _stream(stream)))
    return idx, gate, pred


def mcft_stack_destroy(stack: Stack):
    if stack.handle:
        lib().mcft_stack_destroy(C.c_void_p(stack.handle))
        stack.handle = None


def mcft_cache_tags(cache: Cache, layer, stream=None):
    t = (C.c_int32 * cache.B)()
    _check(lib().mcft_cache_tags(C.c_void_p(cache.handle), layer, C.cast(t, C.c_void_p),
                                 _stream(stream)))
    return list(t)


def mcft_cache_export(cache: Cache, stream=None) -> bytes:
    n = C.c_size_t(0)
    _check(lib().mcft_cache_export(C.c_void_p(cache.handle), None, C.byref(n), _stream(stream)))
    buf = C.create_string_buffer(n.value)
    _check(lib().mcft_cache_export(C.c_void_p(cache.handle), C.cast(buf, C.c_void_p), C.byref(n),
                                   _stream(stream)))
    return buf.raw[: n.value]


def mcft_cache_import(cache: Cache, state: bytes, stream=None):
    buf = C.create_string_buffer(state, len(state))
    _check(lib().mcft_cache_import(C.c_void_p(cache.handle), C.cast(buf, C.c_void_p), len(state),
                                   _stream(stream)))


def mcft_test_inject(fail_pinned_allocs=0, fail_expert_copies=0, wait_limit_ns=0,
                     withhold_gemm13=False):
    """Failure injection for tests (all zero: normal operation)."""
    _check(lib().mcft_test_inject(int(fail_pinned_allocs), int(fail_expert_copies),
                                  int(wait_limit_ns), 1 if withhold_gemm13 else 0))


MCFT_TC_TILES_ONE_CTA, MCFT_TC_TILES_CTA_PAIR = 0, 1


def mcft_set_tc_tiles(mode: int):
    """Expert-GEMM tile shape for the tensor-core forward (process-wide; set before sizing
    workspaces): MCFT_TC_TILES_ONE_CTA (default) or MCFT_TC_TILES_CTA_PAIR."""
    _check(lib().mcft_set_tc_tiles(int(mode)))


def mcft_profile_enable(on: bool = True):
    _check(lib().mcft_profile_enable(1 if on else 0))


def mcft_profile_reset():
    _check(lib().mcft_profile_reset())


def mcft_profile_read():
    """{kernel name: (launches, total ms)} since the last reset (synchronises recorded events)."""
    n = C.c_int(0)
    _check(lib().mcft_profile_read(0, None, None, None, C.byref(n)))
    names = (C.c_char_p * n.value)()
    launches = (C.c_uint64 * n.value)()
    ms = (C.c_double * n.value)()
    _check(lib().mcft_profile_read(n.value, C.cast(names, C.c_void_p), C.cast(launches, C.c_void_p),
                                   C.cast(ms, C.c_void_p), C.byref(n)))
    return {names[i].decode(): (launches[i], ms[i]) for i in range(n.value)}


def mcft_mask_sample(m_tilde, uniforms, e_keep, stream=None):
    """(mask [L, E] uint8, pi [L, E] fp32) from m~ and uniforms [L, E] (device tensors)."""
    L, E = m_tilde.shape
    mask = torch.empty((L, E), dtype=torch.uint8, device=m_tilde.device)
    pi = torch.empty((L, E), dtype=torch.float32, device=m_tilde.device)
    _check(lib().mcft_mask_sample(_ptr(m_tilde), _ptr(uniforms), L, E, int(e_keep), _ptr(mask),
                                  _ptr(pi), _stream(stream)))
    return mask, pi


def mcft_gate_grad(desc: LayerDesc, dy, workspace, dgate=None, stream=None):
    """dL/dg [T, K] from dL/dy and the workspace of the forward of the same batch."""
    T = dy.shape[0]
    if dgate is None:
        dgate = torch.empty((T, desc.K), dtype=torch.float32, device=dy.device)
    _check(lib().mcft_gate_grad(C.byref(desc), _ptr(dy), T, _ptr(workspace), workspace.numel(),
                                _ptr(dgate), _stream(stream)))
    return dgate


def mcft_mask_grad(desc: LayerDesc, idx, gate, dgate, pi, dm=None, dm_tilde=None, accumulate=False,
                   stream=None):
    """(dL/dm [E], dL/dm~ [E]) of one layer (straight-through estimator, Eq. ste)."""
    T = idx.shape[0]
    if dm is None:
        dm = torch.empty(desc.E, dtype=torch.float32, device=idx.device)
    if dm_tilde is None:
        dm_tilde = torch.zeros(desc.E, dtype=torch.float32, device=idx.device)
    _check(lib().mcft_mask_grad(C.byref(desc), _ptr(idx), _ptr(gate), _ptr(dgate), T, _ptr(pi),
                                _ptr(dm), _ptr(dm_tilde), 1 if accumulate else 0, _stream(stream)))
    return dm, dm_tilde
