/*
 * mcft.h - C ABI of libmcft: the masked MoE layer forward and the per-layer expert cache, on one
 * NVIDIA GB300 (sm_103a).
 *
 * The method (MaskCoFT, arxiv 2609.34077) restricts or re-ranks the Top-K routing of each MoE layer
 * with a per-layer mask, so that decoding touches fewer experts and an expert cache in GPU memory
 * misses less often. This library computes, per layer:
 *
 *   z = W x,  p = softmax(z)                                   (Section 3.1)
 *   A = TopK(p)            plain routing                        (Section 3.1, Eq. topk)
 *   A = TopK(p * m)        hard binary mask, fine-tuning        (Section 3.2, Eq. stage1)
 *   A = TopK(p * pi)       soft prior, inference                (Section 3.2, Eq. inference)
 *   y = sum_{i in A} g_i F_i(x)  (+ shared experts)             (Section 3.1, Eq. topk)
 *
 * with g_i from p (renormalised over A for Mixtral, p_i for DeepSeek), F_i a SwiGLU expert, and the
 * per-layer cache of B experts of Section 4.1 ("Simulation", LRU / LFU / FIFO replacement): misses
 * counted per Eq. metrics and fetched from pinned host memory.
 *
 * Conventions for every call:
 *  - Device pointers are caller-owned CUDA device memory; host pointers are caller-owned host
 *    memory read (or written) before the call returns, unless stated otherwise.
 *  - Calls are asynchronous on the given stream unless stated otherwise; a NULL stream is the
 *    legacy default stream.
 *  - Argument errors are found on the host and returned synchronously as MCFT_ERR_INVALID (or
 *    MCFT_ERR_UNSUPPORTED for shapes the library does not handle); nothing is launched then.
 *  - Errors found inside a kernel (an expert id out of range, a missing expert pointer, a wait that
 *    ran out of time) set a device error word and make the remaining kernels of that call skip
 *    their work; mcft_device_error() reads and clears it.
 *  - No call throws; mcft_last_error() returns a message for the calling thread's last error.
 *  - The library keeps, per device, the device addresses of its own static device arrays (the
 *    error word, the scratch of mcft_moe_forward_noalloc), looked up on first use. A
 *    cudaDeviceReset() destroys the context those addresses belong to: after one, no mcft call may
 *    be made on that device in the same process, and handles created before it are invalid.
 *  - Layouts are row-major. dtype MCFT_BF16 means bf16 x, weights and y (fp32 accumulation);
 *    MCFT_F32 means fp32 everywhere (CUDA-core arithmetic, no TF32).
 */
#ifndef MCFT_H
#define MCFT_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Same type as cudaStream_t, declared here so that this header needs no CUDA header. */
typedef struct CUstream_st* mcft_stream_t;

typedef enum {
  MCFT_OK = 0,
  MCFT_ERR_INVALID = 1,      /* bad argument (found on the host) or bad data (found on device) */
  MCFT_ERR_OOM = 2,          /* a device or pinned host allocation failed */
  MCFT_ERR_CUDA = 3,         /* a CUDA runtime call failed; mcft_last_error() has the text */
  MCFT_ERR_TIMEOUT = 4,      /* a kernel's bounded wait ran out; the kernel returned early */
  MCFT_ERR_UNSUPPORTED = 5   /* valid but outside what the library handles (e.g. E > 64) */
} mcft_status;

/* Routing rule. Section 3.1 Eq. topk / Section 3.2 Eq. stage1 / Section 3.2 Eq. inference. */
typedef enum {
  MCFT_ROUTE_TOPK = 0,        /* A = TopK(p) */
  MCFT_ROUTE_HARD_MASK = 1,   /* A = TopK(p * m): only experts with m_e = 1 are eligible */
  MCFT_ROUTE_SOFT_PRIOR = 2   /* A = TopK(p * pi), pi > 0: every expert stays eligible */
} mcft_route_mode;

/* Gate weights, always from p (Section 3.1, text after Eq. topk; Section 3.2 after Eq. inference). */
typedef enum {
  MCFT_GATE_RENORM = 0,  /* Mixtral:  g_i = p_i / sum_{j in A} p_j */
  MCFT_GATE_PLAIN = 1    /* DeepSeek: g_i = p_i                      */
} mcft_gate_mode;

typedef enum { MCFT_F32 = 0, MCFT_BF16 = 1 } mcft_dtype;

/* Shape of one MoE layer (Section 3.1; model sizes of Appendix A Table 4).
 *   d        hidden size d_h; multiple of 64
 *   E        routed experts, 1..64
 *   K        active experts per token, 1..min(E, 8)
 *   w        SwiGLU width of every expert (routed and shared); multiple of 64
 *   n_shared shared experts (DeepSeek-V2-Lite: 2), each of width w, added un-gated, 0..8
 *   gate     mcft_gate_mode
 *   dtype    mcft_dtype of x, router and expert weights, and y */
typedef struct {
  int d, E, K, w, n_shared, gate, dtype;
} mcft_layer_desc;

/* Packed expert block: one contiguous allocation per expert, [W1 | W3 | W2] with
 * W1, W3 of shape [w, d] (gate and up projections) and W2 of shape [d, w] (down projection),
 * so that F(x) = W2 (silu(W1 x) * (W3 x)). Size: 3 * w * d elements of the layer dtype. One
 * block is one unit of cache traffic (one copy per fetch). Base address 16-byte aligned. */

/* ---------------------------------------------------------------------------------------------
 * mcft_route: router GEMV/GEMM, mask or prior, Top-K, softmax gates.
 * Section 3.1 (z = W x, p = softmax(z), Eq. topk), Section 3.2 Eq. stage1 (hard mask) and
 * Eq. inference (soft prior); gate weights from p.
 *
 *   x        device [T, d], layer dtype
 *   T        tokens, >= 0 (T = 0 is a no-op)
 *   w_router device [E, d], layer dtype
 *   mode     mcft_route_mode
 *   mask     host [E] bytes, 0 or 1, at least K ones; read only in HARD_MASK mode (else may be NULL)
 *   prior    host [E] fp32, every entry > 0 and finite; read only in SOFT_PRIOR mode
 *   idx      device [T, K] int32 out: active experts, by descending score; equal scores go to the
 *            lower expert index. SOFT_PRIOR ranks by z_e + log(pi_e), which orders experts exactly
 *            as p_e * pi_e does.
 *   gate     device [T, K] fp32 out: gate weight of each active expert
 * Errors: MCFT_ERR_INVALID for a NULL pointer, bad desc, a mask with fewer than K ones, a prior
 * entry <= 0 or not finite; MCFT_ERR_UNSUPPORTED for E > 64 or K > 8. */
mcft_status mcft_route(const mcft_layer_desc* desc, const void* x, int T, const void* w_router,
                       int mode, const uint8_t* mask, const float* prior, int32_t* idx, float* gate,
                       mcft_stream_t stream);

/* ---------------------------------------------------------------------------------------------
 * mcft_moe_workspace_size: bytes of device workspace mcft_moe_forward needs for up to T_max
 * tokens of this layer shape. */
mcft_status mcft_moe_workspace_size(const mcft_layer_desc* desc, int T_max, size_t* bytes);

/* mcft_moe_forward: token permutation by expert, grouped SwiGLU expert FFN, weighted combine and
 * shared experts: y[t] = sum_k gate[t,k] F_{idx[t,k]}(x[t]) + sum_s F^shared_s(x[t]).
 * Section 3.1 Eq. topk (and the shared experts described after it).
 *
 *   x         device [T, d] layer dtype
 *   idx, gate device [T, K] as written by mcft_route (any ids in [0, E) are accepted; an id out
 *             of range sets the device error word and the call writes nothing to y)
 *   experts   host array [E] of device pointers to packed expert blocks; an entry may be NULL if
 *             no token of this call selects that expert (a NULL that is selected sets the device
 *             error word). The array itself is read before the call returns.
 *   shared    host array [n_shared] of device pointers to packed blocks (NULL if n_shared = 0)
 *   y         device [T, d] layer dtype out (may not alias x)
 *   workspace device, at least mcft_moe_workspace_size(desc, T) bytes, 256-byte aligned; used
 *             by the call's kernels until they finish on the stream
 * bf16 layers with T > 64 tokens run the expert GEMMs on tcgen05 tensor cores (TMA-fed, fp32
 * accumulators in tensor memory, SiLU*up fused in the epilogue, hidden activation rounded to bf16);
 * smaller bf16 batches run an HBM-streaming GEMV; fp32 layers run CUDA-core fp32 arithmetic.
 * Errors: MCFT_ERR_INVALID for a NULL pointer, bad desc, workspace too small or misaligned. */
mcft_status mcft_moe_forward(const mcft_layer_desc* desc, const void* x, int T, const int32_t* idx,
                             const float* gate, const void* const* experts,
                             const void* const* shared, void* y, void* workspace, size_t ws_bytes,
                             mcft_stream_t stream);

/* mcft_moe_forward_lora / mcft_moe_workspace_size_lora: the same layer forward with LoRA
 * adapters on the experts, the Stage-2 co-adaptation forward (Section 3.2: routers and experts are
 * fine-tuned under the fixed mask, the experts through LoRA; Appendix B: rank 8, alpha 16). Each
 * projection of an adapted expert becomes W v + s B (A v), s = lora_scale (alpha / rank):
 *   F(x) = (W2 + s B2 A2) (silu((W1 + s B1 A1) x) * ((W3 + s B3 A3) x)).
 *   expert_lora  host array [E] of device pointers to packed adapter blocks, NULL for an expert
 *                without an adapter; block layout (layer dtype, row-major), r = lora_rank:
 *                [A1 (r x d) | B1 (w x r) | A3 (r x d) | B3 (w x r) | A2 (r x w) | B2 (d x r)],
 *                3 r (d + w) elements, 16-byte aligned
 *   shared_lora  host array [n_shared], same layout (NULL entries allowed; NULL if n_shared = 0)
 *   lora_rank    8 or 16 (MCFT_ERR_UNSUPPORTED otherwise); lora_scale finite
 * The workspace needs mcft_moe_workspace_size_lora(desc, lora_rank, T) bytes. On the tensor-core
 * path (bf16, T > 64) the down projections are skinny GEMMs on the tensor cores and the up
 * projections one extra k-block of each adapted tile of the expert GEMMs; on the decode and fp32
 * paths a small kernel computes A v and the up projections are added as the expert GEMV finishes
 * each output. Adapters that add nothing (B = 0, or none) give mcft_moe_forward's result bit for
 * bit. No dropout (a forward whose output is compared). */
mcft_status mcft_moe_workspace_size_lora(const mcft_layer_desc* desc, int lora_rank, int T_max,
                                         size_t* bytes);
mcft_status mcft_moe_forward_lora(const mcft_layer_desc* desc, const void* x, int T,
                                  const int32_t* idx, const float* gate,
                                  const void* const* experts, const void* const* shared,
                                  const void* const* expert_lora, const void* const* shared_lora,
                                  int lora_rank, float lora_scale, void* y, void* workspace,
                                  size_t ws_bytes, mcft_stream_t stream);

/* mcft_moe_forward_noalloc: the same computation as mcft_moe_forward (same arguments, minus the
 * workspace), for callers that cannot allocate device memory when they run a layer, such as a
 * plugin inside an application that owns every device allocation, or a decode loop that cannot
 * afford an allocation's implicit synchronisation. The paper has no counterpart: this is an
 * interface for such callers only. Scratch comes from one static device array of 16 MiB inside
 * the library (held by every GPU that loads it, until exit), enough for decode calls of up to 64
 * tokens of the Mixtral- and DeepSeek-V2-Lite-shaped layers; a call needing more returns
 * MCFT_ERR_UNSUPPORTED (use mcft_moe_forward). The first call on a device looks up the array's
 * device address; make it before any stream capture. The address is kept for the life of the
 * process, so after a cudaDeviceReset() this entry point must not be called on that device again.
 * All calls share the array: calls whose kernels overlap on the GPU race and must be serialised by
 * the caller. Allocates nothing. */
mcft_status mcft_moe_forward_noalloc(const mcft_layer_desc* desc, const void* x, int T,
                                     const int32_t* idx, const float* gate,
                                     const void* const* experts, const void* const* shared,
                                     void* y, mcft_stream_t stream);

/* ---------------------------------------------------------------------------------------------
 * Per-layer expert cache (Section 4.1 "Simulation"; Eq. metrics).
 * L layers, each with B slots for routed experts, K <= B < E. Caches start empty and persist
 * across calls; first fills count as misses. Per layer and decode step t:
 *   U = distinct experts selected by the step's tokens, each counting one access; cached experts
 *   of U are hits and get last_use = t; the others are misses, one fetch each, taken in ascending
 *   expert id: a miss takes the lowest free slot, else evicts, among slots not used at step t, the
 *   one with the smallest policy key
 *     LRU  (last_use, expert id)
 *     LFU  (accesses of the expert since the stream began, last_use, expert id)
 *     FIFO (step the expert was inserted, expert id);
 *   if every slot was used at step t (possible only when |U| > B) the expert is fetched into a
 *   staging buffer for this step only ("bypass") and not cached.
 *   At batch size 1 this is the paper's cache and f = K - h.
 * Shared experts are not cached here (always resident, Section 4.1). */
typedef struct mcft_cache mcft_cache;

/* Replacement policy (Section 4.1: LRU, LFU, FIFO; Table 2). */
typedef enum { MCFT_CACHE_LRU = 0, MCFT_CACHE_LFU = 1, MCFT_CACHE_FIFO = 2 } mcft_cache_policy;

/* mcft_cache_create: allocate the device tag/timestamp/counter arrays, L*B device slots of
 * expert_bytes each, and the bypass staging buffers (min(E - B, max_assign) of them).
 *   host_experts  host array [L*E] of pinned host pointers to packed expert blocks (layer-major),
 *                 read during the call and kept; the blocks themselves must stay valid and
 *                 pinned until mcft_cache_destroy. NULL = accounting only: no slots are
 *                 allocated and mcft_fetch_experts copies nothing.
 *   max_assign    largest T*K any mcft_cache_step call will pass.
 *   policy        mcft_cache_policy.
 * Synchronous. Errors: MCFT_ERR_INVALID (B < 1, B >= E, E > 64, unknown policy, ...), MCFT_ERR_OOM. */
mcft_status mcft_cache_create(int L, int E, int B, size_t expert_bytes,
                              const void* const* host_experts, int max_assign, int policy,
                              mcft_cache** out);

/* mcft_cache_step: one decode step of one layer. Reads idx (device [T, K] int32), drops the
 * experts the layer's last prefetch loaded that this step does not use (mcft_cache_prefetch),
 * decides hits, misses, evictions and bypasses on the device, updates the counters and writes the
 * step's miss list to host-mapped memory for mcft_fetch_experts. Asynchronous on `stream`.
 * Errors: MCFT_ERR_INVALID (layer out of range, T*K > max_assign, NULL idx); an id out of range
 * sets the device error word and the step changes no state. */
mcft_status mcft_cache_step(mcft_cache* cache, int layer, const int32_t* idx, int T, int K,
                            mcft_stream_t stream);

/* mcft_fetch_experts: complete the last mcft_cache_step of `layer`. The host waits until that
 * step's miss list is written (the fetch cannot start before routing is known), issues one
 * host-to-device copy per missed expert on `copy_stream` (from the pinned host block into its slot
 * or staging buffer), and makes `compute_stream` wait for those copies. Writes, into the host
 * array expert_ptrs [E], the device address of every expert the step selected (NULL for the
 * others), ready to pass to mcft_moe_forward on compute_stream. In accounting mode the addresses
 * are NULL and nothing is copied. Blocks the calling thread until the miss list is known. */
mcft_status mcft_fetch_experts(mcft_cache* cache, int layer, mcft_stream_t compute_stream,
                               mcft_stream_t copy_stream, const void** expert_ptrs);

/* mcft_host_copy: copy `bytes` from pinned host memory to device memory with the device-driven
 * fetch's copy loop (64 KB pieces, 16-byte loads, four in flight per thread) on a grid of `blocks`
 * CTAs of 256 threads. The paper has no counterpart: offloaded decoding is bound by this host link
 * (Section 1), and this call measures what SM loads get from it at a chosen grid size, beside the
 * copy engines. host_src: host memory the device can address (pinned memory, or any host memory
 * on a system whose GPU reads pageable memory, such as a Grace-based node); dst: device memory;
 * both 16-byte aligned; bytes a multiple of 16; 1 <= blocks <= 65535. MCFT_ERR_INVALID for a
 * pointer that is NULL or misaligned, for a host_src the device cannot address, for
 * bytes % 16 != 0 or a bad block count. Asynchronous on `stream`. */
mcft_status mcft_host_copy(void* dst, const void* host_src, size_t bytes, int blocks,
                           mcft_stream_t stream);

/* mcft_read_probe: read `bytes` of device memory in one launch of `blocks` CTAs of 256 threads,
 * with no computation on the data, to measure what a launch of the decode FFN's shape reads at
 * all (no counterpart in the paper; the decode FFN of Section 3.1's experts streams the selected
 * experts' weights once). pattern 0: one contiguous stream, grid-strided, eight 16-byte loads in
 * flight per thread. pattern 1: exactly the decode FFN's weight loads: items of 32 rows of
 * row_bytes (16 W1 rows, then 16 W3 rows) strided over the grid; warp w of a CTA reads the
 * 128-byte chunks w, w + 8, ... of every row of its item, eight 16-byte loads per lane per step.
 * Every 32-bit word is read once; *sink is XORed with the XOR of all of them (so it equals the
 * buffer's XOR if it started at 0).
 *   buf  device memory, 16-byte aligned; bytes a multiple of 16 (pattern 0) or of 32 * row_bytes
 *        (pattern 1, row_bytes a positive multiple of 128); sink device, one unsigned;
 *   1 <= blocks <= 65535. MCFT_ERR_INVALID otherwise. Asynchronous on `stream`. */
mcft_status mcft_read_probe(const void* buf, size_t bytes, int pattern, int row_bytes, int blocks,
                            unsigned* sink, mcft_stream_t stream);

/* ---------------------------------------------------------------------------------------------
 * Stage-1 mask machinery (Section 3.2 "Stage 1" Eq. stage1 and "Mask optimization" Eq. ste).
 *
 * mcft_mask_sample: per layer l, pi_l = softmax(m~_l) and a binary mask with exactly e_keep ones:
 * E' = e_keep experts drawn without replacement from pi_l (MultinomialSample), realised by the
 * Gumbel-top-k rule with caller-drawn uniforms: key_e = log pi_e - log(-log u_e); the e_keep
 * largest keys are drawn (ties to the lower index). This has the law of sequential draws without
 * replacement. All pointers device: m_tilde, uniforms [L, E] fp32 (uniforms in (0, 1); one
 * outside sets the device error word and that expert is never drawn), mask [L, E] bytes out,
 * pi [L, E] fp32 out. 1 <= e_keep <= E <= 64. */
mcft_status mcft_mask_sample(const float* m_tilde, const float* uniforms, int L, int E, int e_keep,
                             uint8_t* mask, float* pi, mcft_stream_t stream);

/* mcft_gate_grad: dL/dg_{t,k} = < dL/dy_t , F_{idx[t,k]}(x_t) > for the batch of the last
 * mcft_moe_forward (or _lora, _cached) call that used `workspace` with this desc and T: the expert
 * outputs are read from that workspace, which must be left untouched in between.
 *   dy device [T, d] layer dtype (gradient of the loss with respect to y); dgate device [T, K]
 *   fp32 out. */
mcft_status mcft_gate_grad(const mcft_layer_desc* desc, const void* dy, int T, const void* workspace,
                           size_t ws_bytes, float* dgate, mcft_stream_t stream);

/* mcft_mask_grad: the straight-through mask gradient of one layer (Eq. ste). The loss reaches m
 * through the gates of the active experts, computed from p * m with m = 1 on A: renormalised gates
 * (Mixtral) give dL/dm_e = sum_{t: e in A_t} g_{t,e} (dL/dg_{t,e} - sum_i g_{t,i} dL/dg_{t,i}),
 * plain gates (DeepSeek) dL/dm_e = sum_{t: e in A_t} g_{t,e} dL/dg_{t,e}; the sum runs over every
 * token of the batch (deterministic order). Then dL/dm~ = (diag(pi) - pi pi^T) dL/dm.
 *   idx, gate, dgate device [T, K]; pi device [E]; dm device [E] out; dm_tilde device [E] out,
 *   or accumulated into when `accumulate` is non-zero (the paper accumulates the mask gradient
 *   over several steps before one update). */
mcft_status mcft_mask_grad(const mcft_layer_desc* desc, const int32_t* idx, const float* gate,
                           const float* dgate, int T, const float* pi, float* dm, float* dm_tilde,
                           int accumulate, mcft_stream_t stream);

/* mcft_moe_forward_cached: mcft_moe_forward for a decode step of `layer` whose experts come from
 * the cache, with the fetch driven by the device and overlapped with compute; no host round trip.
 * Call it once after each mcft_cache_step(cache, layer, idx, ...) on compute_stream, instead of
 * mcft_fetch_experts + mcft_moe_forward (the fetching launch below claims its copy work from
 * counters that cache step resets). Every missed expert's block is copied from pinned host
 * memory into the slot or staging buffer the cache step chose, by SM loads over the host link:
 *  - bf16, T <= 16, and no prefetch of any layer in flight: in the FFN's own launch on
 *    compute_stream, whose first CTAs copy the misses piece by piece while the others compute the
 *    hits (and shared experts); a missed expert's work items start as the pieces they read land,
 *    so its FFN runs while the rest of the step's bytes are still on the host link (copy_stream is
 *    not used);
 *  - otherwise: on copy_stream (after that cache step) a fetch kernel copies them while the
 *    permutation and the FFN of the hits run on compute_stream; then compute_stream waits for the
 *    copies and computes the fetched experts.
 * Then the combine. Results equal mcft_moe_forward's with the same experts, bit for bit (a decode
 * work item has the same shape and summation order whichever launch computes its expert).
 * Section 3.1 Eq. topk (the layer); Section 1 and Section 3.1 "Preliminaries" (every miss is a fetch
 * from host memory).
 *   cache  created with host blocks (not accounting-only); its E and expert size match desc
 *   other arguments as for mcft_moe_forward (the routed expert addresses come from the cache)
 * Supports the decode path (bf16 with T <= 64, or fp32); larger bf16 calls return
 * MCFT_ERR_UNSUPPORTED (use mcft_fetch_experts + mcft_moe_forward). Asynchronous. */
mcft_status mcft_moe_forward_cached(const mcft_layer_desc* desc, const void* x, int T,
                                    const int32_t* idx, const float* gate, mcft_cache* cache,
                                    int layer, const void* const* shared, void* y, void* workspace,
                                    size_t ws_bytes, mcft_stream_t compute_stream,
                                    mcft_stream_t copy_stream);

/* mcft_cache_prefetch: a prefetch event of `layer` (no counterpart rule in the paper; offloading
 * systems load experts ahead of need, Section 2 "Offloading systems for MoE inference"). From the
 * predicted routing idx_pred (device [T, K] int32, each row in descending score, e.g. mcft_route
 * of the layer's router on a speculative input) the candidates are the experts it names, ranked by
 * how many predictions name them, then the best rank k at which a token predicts them, then the
 * lower id. Every cached candidate is touched (last use = this event, which has a time stamp of
 * its own between two steps; no LFU access is counted), so this event evicts none of them; the
 * n_max best-ranked uncached candidates, in ascending id, take the lowest free slot or evict,
 * among slots not touched at this event, the smallest policy key (skipped if none qualifies).
 * Each load counts as one prefetched expert; a prefetched expert that the layer's next
 * mcft_cache_step uses counts as useful, one it does not use is dropped by that step (its slot
 * becomes free before the step's hits and misses) and the prefetch's fetch stops copying it.
 * Decided on the device on `stream`.
 * The loads are fetched (device-driven, host link) on the copy stream of the next
 * mcft_moe_forward_cached or mcft_fetch_experts call on this cache, behind that call's own misses
 * (or, for this layer, before them). The layer's next step treats experts still arriving from
 * the prefetch like its misses: mcft_moe_forward_cached computes them after its copies,
 * mcft_fetch_experts makes compute_stream wait for them. All calls on one cache must use one copy
 * stream.
 *   1 <= n_max <= B; T*K <= max_assign.
 * Errors: MCFT_ERR_INVALID (bad arguments; a previous prefetch of the layer not yet fetched);
 * MCFT_ERR_UNSUPPORTED (host blocks without device-visible addresses); an id out of range sets the
 * device error word and changes no state. Accounting-only caches record the decision only. */
mcft_status mcft_cache_prefetch(mcft_cache* cache, int layer, const int32_t* idx_pred, int T, int K,
                                int n_max, mcft_stream_t stream);

/* mcft_cache_prefetch_stats: cumulative prefetched experts, useful prefetches (prefetched
 * experts used by the next step) and bytes the prefetch fetches actually copied (a dropped
 * prefetch stops early) of one layer, or summed when layer = -1. The counts are decisions and
 * exact; bytes_moved depends on timing. Synchronises `stream` first. */
mcft_status mcft_cache_prefetch_stats(const mcft_cache* cache, int layer, uint64_t* prefetched,
                                      uint64_t* useful, uint64_t* bytes_moved, mcft_stream_t stream);

/* mcft_cache_last_misses: the miss list of the last mcft_cache_step of `layer`, after
 * mcft_fetch_experts (or a synchronisation of its stream): n_out = number of fetches;
 * experts[i], slots[i] for i < n_out in processing order, slot = -1 for a bypass fetch.
 * Arrays are host [E]. */
mcft_status mcft_cache_last_misses(const mcft_cache* cache, int layer, int* n_out, int32_t* experts,
                                   int32_t* slots);

/* mcft_cache_stats: cumulative hits, fetches (misses, bypasses included) and bypasses of one
 * layer, or summed over all layers when layer = -1. Synchronises `stream` first. HR and
 * Fetches/tok of Eq. metrics follow as hits / (hits + fetches) and fetches / tokens. */
mcft_status mcft_cache_stats(const mcft_cache* cache, int layer, uint64_t* hits, uint64_t* fetches,
                             uint64_t* bypass, mcft_stream_t stream);

/* mcft_cache_tags: host [B] copy of the expert id held by each slot of `layer` (-1 = empty).
 * Synchronises `stream` first. */
mcft_status mcft_cache_tags(const mcft_cache* cache, int layer, int32_t* tags, mcft_stream_t stream);

/* mcft_cache_export / mcft_cache_import: checkpoint of the whole cache state (tags, last-use and
 * insertion steps, access counts, step counters, counters, pending prefetch set); call them with no
 * prefetch awaiting its fetch. Import into a cache created with the
 * same L, E, B and policy resumes a stream
 * with identical decisions. Slot contents are not part of the state: after an import, the slots
 * the tags name must be refilled by the caller (or the cache used in accounting mode).
 * export with buf = NULL writes the needed size to *bytes. Both synchronise `stream`. */
mcft_status mcft_cache_export(const mcft_cache* cache, void* buf, size_t* bytes, mcft_stream_t stream);
mcft_status mcft_cache_import(mcft_cache* cache, const void* buf, size_t bytes, mcft_stream_t stream);

/* mcft_cache_destroy: free everything mcft_cache_create allocated (synchronises the device). */
void mcft_cache_destroy(mcft_cache* cache);

/* ---------------------------------------------------------------------------------------------
 * Chained decode stack: the residual stream between MoE blocks.
 *
 * mcft_residual_rmsnorm: for each of the T rows, x <- x + y (when y is not NULL), then
 * u = gamma * x / sqrt(mean_j x[j]^2 + eps) (when gamma is not NULL): the block-input RMSNorm of the
 * paper's models (Mixtral-8x7B, DeepSeek-V2-Lite; Section 4, Table 4), which the paper uses but
 * does not restate; eps is 1e-5 for Mixtral, 1e-6 for DeepSeek-V2-Lite. Without attention blocks a
 * decode step of an L-layer stack is u_0 = RMSNorm_0(x_0); for each layer l: route u_l, run the
 * layer on u_l into y_l, then x_{l+1} = x_l + y_l and u_{l+1} = RMSNorm_{l+1}(x_{l+1}) (one call).
 *   x      device [T, d] fp32 residual stream, updated in place when y is given
 *   y      device [T, d] layer dtype, or NULL
 *   gamma  device [d] layer dtype, or NULL (then u is not written)
 *   u      device [T, d] layer dtype out (bf16: rounded to nearest even)
 * All pointers 16-byte aligned; 0 <= eps <= 1. One CTA per row; the sum of squares is reduced in a
 * fixed order (deterministic). Asynchronous on `stream`. */
mcft_status mcft_residual_rmsnorm(const mcft_layer_desc* desc, float* x, const void* y, int T,
                                  const void* gamma, float eps, void* u, mcft_stream_t stream);

/* mcft_stack_create: an L-layer chained decode stack on the residual stream (no counterpart API in
 * the paper; its models are such stacks with attention blocks in between, which this library does
 * not have). Each step runs, per layer l: RMSNorm_l, soft-prior routing (Section 3.2 Eq. inference)
 * by layer l's router, the cache step of layer l, optionally the prefetch event of layer l+1 from
 * the routing of RMSNorm_{l+1}(x_l) by layer l+1 (the stream before layer l's output is added),
 * mcft_moe_forward_cached of layer l, and x <- x + y. No host synchronisation: a step can be
 * captured in a CUDA graph.
 *   routers    host [L] device pointers to router weights [E, d] (layer dtype)
 *   priors     host [L*E] fp32 soft priors, every entry > 0 and finite (copied)
 *   gammas     host [L] device pointers to RMSNorm scales [d] (layer dtype)
 *   shared     host [L*S] device pointers to shared expert blocks (NULL when S = 0)
 *   eps        RMSNorm epsilon in [0, 1]
 *   cache      created with L layers, desc's E and expert size, host blocks with device-visible
 *              addresses; used by this stack's steps only while they run
 *   n_prefetch 0 = no prefetch, else the n_max of mcft_cache_prefetch (1 <= n_prefetch <= B)
 *   T_max      largest batch of a step (at most 64 for bf16)
 * The pointed-to weights stay owned by the caller and must outlive the stack. Allocates the
 * stack's activations, routing buffers and one workspace. Synchronous. */
typedef struct mcft_stack mcft_stack;
mcft_status mcft_stack_create(const mcft_layer_desc* desc, int L, const void* const* routers,
                              const float* priors, const void* const* gammas,
                              const void* const* shared, float eps, mcft_cache* cache,
                              int n_prefetch, int T_max, mcft_stack** out);

/* mcft_stack_step: one decode step of all L layers for T tokens (1 <= T <= T_max).
 *   x  device [T, d] fp32: the stream entering layer 0 on input, leaving layer L-1 on output.
 * Kernels on compute_stream, expert fetches on copy_stream. Asynchronous. */
mcft_status mcft_stack_step(mcft_stack* stack, float* x, int T, mcft_stream_t compute_stream,
                            mcft_stream_t copy_stream);

/* mcft_stack_routing: host copies of layer `layer`'s routing in the last step: idx and gate
 * [T, K], and idx_pred [T, K], the prediction made for this layer during the previous layer
 * (valid for layer >= 1 with prefetch on; -1 otherwise). Any pointer may be NULL. Synchronises
 * `stream` after the copies. */
mcft_status mcft_stack_routing(const mcft_stack* stack, int layer, int32_t* idx, float* gate,
                               int32_t* idx_pred, mcft_stream_t stream);

/* mcft_stack_destroy: synchronise the device and free what mcft_stack_create allocated. */
void mcft_stack_destroy(mcft_stack* stack);

/* ---------------------------------------------------------------------------------------------
 * mcft_device_error: synchronise `stream`, return and clear the device error word of the current
 * device: MCFT_OK, MCFT_ERR_INVALID (bad id, missing expert pointer) or MCFT_ERR_TIMEOUT. */
mcft_status mcft_device_error(mcft_stream_t stream);

/* ---------------------------------------------------------------------------------------------
 * Failure injection for tests (no counterpart in the paper). Sets, for the whole process:
 *   fail_pinned_allocs   the next n pinned host allocations of the library fail as if the runtime
 *                        were out of memory (mcft_cache_create then returns MCFT_ERR_OOM and
 *                        frees everything it had allocated);
 *   fail_expert_copies   the next n host-to-device expert copies of mcft_fetch_experts fail as if
 *                        the runtime had refused them (MCFT_ERR_CUDA; the slots that step was
 *                        filling then hold undefined bytes: destroy the cache or import a state);
 *   wait_limit_ns        the limit of the decode FFN's bounded waits (0 = the default, 2 s);
 *   withhold_gemm13      nonzero: the fused decode FFN skips its GEMM13 items, so every GEMM2
 *                        item's wait for its segment runs out after wait_limit_ns; the call then
 *                        sets MCFT_ERR_TIMEOUT in the device error word and leaves y untouched.
 * Nothing here makes a kernel fault or wait without a limit. mcft_test_inject(0, 0, 0, 0) restores
 * normal operation. Not synchronised with calls running on other threads. MCFT_ERR_INVALID for a
 * negative count. */
mcft_status mcft_test_inject(int fail_pinned_allocs, int fail_expert_copies,
                             unsigned long long wait_limit_ns, int withhold_gemm13);

/* ---------------------------------------------------------------------------------------------
 * Tensor-core tile shape of the expert GEMMs (Section 3.1's F(x) for the large-batch forward; no
 * counterpart in the paper: a choice of kernel). Process-wide, read when a call lays out its
 * workspace, so set it before sizing workspaces (mcft_moe_workspace_size) and keep it while they
 * are in use: a workspace sized under one setting may be too small under the other, which the
 * forward then rejects with MCFT_ERR_INVALID.
 *   MCFT_TC_TILES_ONE_CTA   (default) 128 x 256 tiles, one CTA per SM, segments padded to 128
 *                           rows;
 *   MCFT_TC_TILES_CTA_PAIR  256 x 256 tiles on pairs of CTAs (cta_group::2 MMAs issued by one CTA
 *                           of a 2-CTA cluster over both CTAs' shared memory), segments padded to
 *                           256 rows, for layers without adapters whose routed experts average at
 *                           least 512 rows (others keep the one-CTA tiles). Each output is the
 *                           same products summed in the same order; on every shape tested the
 *                           outputs equal the one-CTA tiles' bit for bit. Slower than the one-CTA
 *                           tiles on the GB300 shapes measured (kept for comparison).
 * MCFT_ERR_INVALID for another mode. */
typedef enum { MCFT_TC_TILES_ONE_CTA = 0, MCFT_TC_TILES_CTA_PAIR = 1 } mcft_tc_tiles;
mcft_status mcft_set_tc_tiles(int mode);

/* ---------------------------------------------------------------------------------------------
 * Kernel timing (no counterpart in the paper; used to measure the path). While enabled, every
 * kernel the library launches is bracketed by two CUDA events on its stream.
 * mcft_profile_read synchronises the recorded events and returns, per kernel of the library, its
 * name (static string), launches and total milliseconds since the last mcft_profile_reset;
 * n_out = number of kernels (arrays are host [max]). Not thread-safe against concurrent enabling. */
mcft_status mcft_profile_enable(int on);
mcft_status mcft_profile_reset(void);
mcft_status mcft_profile_read(int max, const char** names, uint64_t* launches, double* ms, int* n_out);

/* mcft_last_error: message for the calling thread's last failed call ("" if none). */
const char* mcft_last_error(void);

/* mcft_version: library version, major * 10000 + minor * 100 + patch. */
int mcft_version(void);

#ifdef __cplusplus
}
#endif

#endif /* MCFT_H */
