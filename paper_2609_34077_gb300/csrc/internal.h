// Internal launchers and the workspace layout shared by the C ABI (api.cu) and the kernels.
#pragma once

#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

#include <utility>

#include <nvtx3/nvToolsExt.h>

#include "../../include/mcft.h"
#include "common.cuh"

namespace mcft {

// NVTX range around a C-ABI call, so timeline profilers show route / cache step / fetch / forward /
// stack step by name (header-only NVTX: nothing happens unless a profiler is attached).
struct NvtxRange {
  explicit NvtxRange(const char* name) { nvtxRangePushA(name); }
  ~NvtxRange() { nvtxRangePop(); }
  NvtxRange(const NvtxRange&) = delete;
  NvtxRange& operator=(const NvtxRange&) = delete;
};

// Launch `kernel` with programmatic stream serialization (programmatic dependent launch): its CTAs
// may be scheduled while the previous kernel in `s` drains, and the kernel's pdl_wait() holds its
// memory accesses until that kernel is complete. Removes most of the launch gap between the small
// dependent kernels of a decode step, also inside a CUDA graph.
template <typename... KArgs, typename... Args>
inline cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem,
                              cudaStream_t s, Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kernel, std::forward<Args>(args)...);
}

struct RouteArgs {
  const void* x;
  const void* w_router;
  int T, d, E, K, mode, gate_mode;
  float prior[64];            // SOFT_PRIOR: pi_e (> 0)
  unsigned char mask[64];     // HARD_MASK: m_e in {0, 1}
  int32_t* idx;
  float* gate;
  unsigned* err;
};
cudaError_t launch_route(const RouteArgs& a, int dtype, cudaStream_t s);
int num_sms();  // SMs of the current device (looked up once per device)
// bf16 calls of more tokens than this route in 16-token tensor-core tiles (route.cu).
constexpr int kRouteTileMinT = 64;

// Header at the start of the forward workspace.
// Work-claim counters of the fused decode FFN that follow the per-segment progress counters in
// the workspace: one per FFN phase (0 all segments, 1 hits, 2 misses).
// slots 0-2: the claim counters of phases 0-2 (the fetching launch's role and piece counters are
// the cache's, FfnArgs::fctr)
constexpr int kClaimSlots = 3;

struct WsHeader {
  int abort;     // set when a kernel of this call found bad data; later kernels skip their work
  int nseg;      // E + n_shared
  int mrows;     // total permuted rows (padded)
  int pad0;
};

// Device workspace of one mcft_moe_forward call. Segments 0..E-1 are the routed experts,
// E..E+S-1 the shared experts (every token). Offsets are in permuted rows.
struct WsLayout {
  int lrank;      // LoRA rank (0: no adapters)
  bool tc;        // tensor-core path (bf16, large T)
  bool decode;    // bf16 decode path (T <= 64)
  int pad;        // rows per segment are padded to a multiple of this (TC path: 128, or 256
                  // for CTA-pair tiles)
  int mcap;       // capacity in permuted rows
  int ks;         // partial planes of o (contraction split of the decode GEMM2)
  size_t hdr, cnt, off, pos, perm, done, pscr, xp, h, o, u13, u2, total;
};
WsLayout ws_layout(int d, int E, int K, int w, int S, int dtype, int T, int lrank = 0);

// LoRA adapter block of one expert (layer dtype, row-major), element offsets for rank r:
// [A1 (r x d) | B1 (w x r) | A3 (r x d) | B3 (w x r) | A2 (r x w) | B2 (d x r)].
struct LoraOffsets {
  size_t a1, b1, a3, b3, a2, b2, total;
};
__host__ __device__ inline LoraOffsets lora_offsets(int d, int w, int r) {
  LoraOffsets o;
  o.a1 = 0;
  o.b1 = size_t(r) * d;
  o.a3 = o.b1 + size_t(w) * r;
  o.b3 = o.a3 + size_t(r) * d;
  o.a2 = o.b3 + size_t(w) * r;
  o.b2 = o.a2 + size_t(r) * w;
  o.total = o.b2 + size_t(d) * r;
  return o;
}

// LoRA down-projection u[q] = A v_q for the permuted rows (lora.cu).
struct LoraDownArgs {
  const void* in;        // input rows: x [T, K] (by token) or h [mcap, K] (by permuted row)
  size_t in_stride;      // elements per input row
  const int* row_tok;    // token of each permuted row, -1 for padding rows
  int by_token;          // 1: input row = row_tok[q]; 0: input row = q
  const int* off;
  const WsHeader* hdr;
  int nseg;
  const void* lblk[72];  // adapter block of each segment (NULL: none)
  size_t a_off0, a_off1; // element offsets of the A matrices used (second only at stage 13)
  int r, K;              // rank, contraction length
  float* u;              // output [mcap, ustride]
  int ustride;
};
cudaError_t launch_lora_down(const LoraDownArgs& a, int dtype, int outs, int mcap, cudaStream_t s);

struct PermuteArgs {
  const int32_t* idx;
  int T, K, E, S, pad, mcap;
  WsHeader* hdr;
  int* cnt;    // [E+S] rows per segment (unpadded)
  int* off;    // [E+S+1] padded segment offsets
  int* pos;    // [T*K] permuted row of assignment (t, k)
  int* perm;   // [mcap] token of each permuted row, -1 for padding
  unsigned* err;
  int* done;   // [E+S + kClaimSlots] progress and claim counters of the fused decode FFN, zeroed here
  int* scr;    // NULL, or kPermScrInts of scratch: large batches then permute in chunks
};
constexpr int kPermChunks = 256;      // most chunks of the large-batch permutation
constexpr int kPermSingleMax = 4096;  // up to this many assignments one CTA permutes (faster)
constexpr int kPermScrInts = kPermChunks * kMaxE + kPermChunks;
cudaError_t launch_permute(const PermuteArgs& a, cudaStream_t s);

struct GatherArgs {
  const void* x;  // [T, d] bf16
  const int* perm;
  const WsHeader* hdr;
  void* xp;       // [mcap, d] bf16
  int d, mcap;
};
cudaError_t launch_gather(const GatherArgs& a, cudaStream_t s);

struct FfnArgs {
  const void* x;                 // [T, d] (FFN13) activations
  const int* off;
  const int* perm;
  const WsHeader* hdr;
  const void* wblk[72];          // packed expert block of each segment
  void* h;                       // [mcap, w] fp32 (rowwise) or bf16 (tensor cores, decode)
  float* o;                      // [ksplit][mcap, d] fp32
  size_t o_plane;                // elements between partial planes of o
  int T, d, w, nseg, E, ksplit;
  unsigned* err;
  // Expert addresses written on the device by a cache step (NULL: use wblk), that step's hit
  // mask, and which segments this launch computes: 0 all, 1 hit experts and shared experts,
  // 2 routed experts that were not hits (fetched or bypassed at this step).
  const unsigned long long* wtab;
  const unsigned long long* ready;
  int phase;
  // LoRA (Stage 2): adapter block of each segment (NULL: none), rank, scale alpha / r, and the
  // down-projections u13 [mcap, 2r] (A1 x, A3 x) and u2 [mcap, r] (A2 h): fp32 from lora_down,
  // or on the tcgen05 path bf16 and scaled by s (s [A1 x | A3 x], s A2 h).
  const void* lblk[72];
  int lrank;
  float lscale;
  const float* u13;
  const float* u2;
  // [E+S] completed GEMM13 items per segment, then kClaimSlots work-claim counters (one per
  // phase), all zeroed by the permutation of the call: they let one fused decode launch hand out
  // its items dynamically and start a segment's GEMM2 as soon as that segment's h is written
  int* done;
  // Limit of the fused decode FFN's bounded waits (ns), and a test switch that makes it skip its
  // GEMM13 items so that those waits run out (set by launch_ffn_decode from the test hooks).
  unsigned long long wait_ns;
  int withhold13;
  // A decode launch that fetches its own misses (cached forward, small bf16 batches, no prefetch
  // in flight): its first nfetch CTAs to start copy the step's missed expert blocks (miss list
  // fmiss, device-visible host blocks fsrc [E], destinations wtab [E], fbytes each) piece by
  // piece, stamping each kFetchPiece-byte piece in landed [E][ppe] with the step's epoch (*epoch,
  // the layer's step count after its cache step) once its bytes are written, then join the FFN.
  // stream has bit e set when expert e is such a miss: the launch computes those experts with the
  // hits, each of their items waiting (bounded) for the pieces it reads, so their FFN runs while
  // the rest of the step's bytes are still on the host link. nfetch = 0: no fetch, no streaming.
  const unsigned long long* stream;
  unsigned* fctr;  // [2] role and piece counters, zeroed by the layer's cache step
  unsigned* landed;
  const int64_t* epoch;
  int ppe;
  const int32_t* fmiss;
  const unsigned long long* fsrc;
  size_t fbytes;
  int nfetch;
};

// Bytes per work unit of the device-driven fetch: the granule of its landed stamps.
constexpr size_t kFetchPiece = 65536;
// Cached decode forwards of up to this many tokens stream their misses behind the fetch.
constexpr int kStreamMaxT = 16;

// Test hooks (mcft_test_inject in api.cu); all off by default.
unsigned long long test_wait_limit_ns();  // the decode FFN's wait limit (default 2 s)
bool test_withhold_gemm13();              // skip the decode FFN's GEMM13 items

// s * sum_j u[j] B[row][j] for a LoRA up-projection B [rows, r] (layer dtype TW).
template <typename TW>
__device__ __forceinline__ float lora_up(const void* blk, size_t b_off, int row, const float* u,
                                         int r, float scale);
template <>
__device__ __forceinline__ float lora_up<__nv_bfloat16>(const void* blk, size_t b_off, int row,
                                                        const float* u, int r, float scale) {
  const char* b = reinterpret_cast<const char*>(blk) + (b_off + size_t(row) * r) * 2;
  float acc = 0.f;
  for (int j = 0; j < r; j += 8) {
    float w8[8];
    unpack8(__ldg(reinterpret_cast<const uint4*>(b + j * 2)), w8);
#pragma unroll
    for (int i = 0; i < 8; ++i) acc = fmaf(u[j + i], w8[i], acc);
  }
  return scale * acc;
}
template <>
__device__ __forceinline__ float lora_up<float>(const void* blk, size_t b_off, int row, const float* u,
                                                int r, float scale) {
  const float* b = reinterpret_cast<const float*>(blk) + b_off + size_t(row) * r;
  float acc = 0.f;
  for (int j = 0; j < r; ++j) acc = fmaf(u[j], __ldg(b + j), acc);
  return scale * acc;
}

// Segment s of a forward: its block address and whether this launch computes it.
__device__ __forceinline__ const void* seg_block(const FfnArgs& a, int s) {
  return (a.wtab && s < a.E) ? reinterpret_cast<const void*>(a.wtab[s]) : a.wblk[s];
}
// Phase 1 computes the hit and shared experts and the experts streamed behind their fetch, phase 2
// the others (experts a prefetch is still bringing in; without streaming, also the misses).
__device__ __forceinline__ bool seg_streamed(const FfnArgs& a, int s, unsigned long long stream) {
  return a.landed != nullptr && s < a.E && ((stream >> s) & 1ull);
}
__device__ __forceinline__ bool seg_in_phase(const FfnArgs& a, int s, unsigned long long hits,
                                             unsigned long long stream = 0) {
  if (a.phase == 0) return true;
  const bool first = s >= a.E || ((hits >> s) & 1ull) || seg_streamed(a, s, stream);
  return a.phase == 1 ? first : !first;
}
// stages: bit 0 = GEMM13 (+ SwiGLU), bit 1 = GEMM2
cudaError_t launch_ffn_rowwise(const FfnArgs& a, int dtype, int num_sms, cudaStream_t s,
                               int stages = 3);  // fp32
// reserved: CTA slots left free for another kernel that may run at the same time (the expert
// fetch, which otherwise could not start until the FFN's CTAs exit).
cudaError_t launch_ffn_decode(const FfnArgs& a, int num_sms, cudaStream_t s, int stages = 3,
                              int reserved = 0);  // bf16, T <= 64
int decode_ksplit(int T);  // contraction split of the decode GEMM2 for T tokens
// pad: rows per segment of the permutation, 128 (one-CTA tiles) or 256 (CTA-pair tiles, which
// tc_pair_tiles chooses for layers without adapters whose routed experts average >= 512 rows).
cudaError_t launch_ffn_tc(const FfnArgs& a, const void* xp, int mcap, int pad, int num_sms,
                          cudaStream_t s, int stages = 3);
bool tc_pair_tiles(int T, int K, int E, int lrank);
// Down projections of the adapters for the tcgen05 path, on the tensor cores, bf16 out scaled by
// s: stage 1: u13[q] = s [A1 xp[q] | A3 xp[q]] (N = 2r); stage 2: u2[q] = s A2 h[q] (N = 16),
// for the rows of every segment with an adapter. The expert GEMMs add the up projections.
cudaError_t launch_lora_down_tc(const FfnArgs& a, const void* xp, int mcap, int num_sms,
                                cudaStream_t s, int stage);

struct CombineArgs {
  const float* o;
  const float* gate;
  const int* pos;
  const int* off;
  const WsHeader* hdr;
  void* y;
  int T, d, K, E, S, ks;  // ks partial planes of o, o_plane elements apart
  size_t o_plane;
};
cudaError_t launch_combine(const CombineArgs& a, int dtype, cudaStream_t s);

// Cache step kernel state (device arrays of one cache).
struct CacheStepArgs {
  const int32_t* idx;
  int n;              // T*K ids
  int E, B, layer, policy;
  int32_t* tag;       // [L*B]
  int64_t* last;      // [L*B] step of last use
  int64_t* ins;       // [L*B] step of insertion (FIFO)
  int64_t* freq;      // [L*E] accesses per expert since the stream began (LFU)
  int64_t* step;      // [L]
  unsigned long long* counters;  // [L*kCacheCounters] hits, fetches, bypass, prefetched, useful
  unsigned long long* pfmask;    // [L] experts loaded by a prefetch since the layer's last step
  unsigned long long* cancel;    // [L] prefetched experts this step dropped (read by the fetch)
  int32_t* miss_out;  // host-mapped, per layer: [n_miss, expert[E], loc[E], loc_of[E]]
  int32_t* miss_dev;  // device copy of the same list (read by the fetch kernel)
  unsigned long long* ptr_tab;  // device [E]: block address of each selected expert, else 0
  unsigned long long* ready;    // device: bit e set when expert e was a hit at this step
  unsigned long long* stream;   // device: bit e set when expert e is a miss of this step (copied
                                // by the step's demand fetch); NULL: not published
  unsigned* fctr;               // device [2]: role and piece counters of the decode FFN launch
                                // that fetches this step's misses, zeroed here; NULL: none
  const char* slots;            // this layer's first slot block (NULL in accounting mode)
  const char* staging;          // bypass staging blocks
  size_t expert_bytes;
  unsigned* err;
};
cudaError_t launch_cache_step(const CacheStepArgs& a, cudaStream_t s);

constexpr int kCacheCounters = 5;  // per layer: hits, fetches, bypass, prefetched, useful

// Prefetch decision of one layer: the experts of the predicted routing that are cached are
// touched, and the n_max best-ranked uncached ones (by count, then best predicted rank, then id)
// are loaded into the layer's slots (cache.cu).
struct PrefetchArgs {
  const int32_t* idx;  // predicted routing [n / K][K], each row in descending score
  int n, K, n_max;
  int E, B, layer, policy;
  int32_t* tag;
  int64_t* last;
  int64_t* ins;
  const int64_t* freq;
  int64_t* step;
  unsigned long long* counters;
  unsigned long long* pfmask;
  unsigned long long* cancel;     // [L]: cleared for the layer by a new prefetch
  int32_t* list;                  // device, this layer: [n_load, expert[E]] (fetch list)
  unsigned long long* ptr_tab;    // device [E]: destination of each loaded expert, else 0
  const char* slots;              // this layer's first slot block (NULL in accounting mode)
  size_t expert_bytes;
  unsigned* err;
};
cudaError_t launch_prefetch(const PrefetchArgs& a, cudaStream_t s);

// Device-driven fetch: copy the blocks of a layer's missed experts from pinned host memory
// (device-visible addresses host_src[E]) into the addresses ptr_tab[E] chosen by the cache step.
struct FetchArgs {
  const int32_t* miss;                // device miss list of the layer [1 + 3E]
  const unsigned long long* host_src; // [E]
  const unsigned long long* ptr_tab;  // [E]
  size_t bytes;                       // per expert block, multiple of 16
  const unsigned long long* cancel;   // prefetch fetches: experts to stop copying, else NULL
  unsigned long long* moved;          // prefetch fetches: bytes copied (accumulated), else NULL
};
cudaError_t launch_fetch(const FetchArgs& a, int blocks, cudaStream_t s, bool prefetch = false);
// Plain copy from device-visible host memory with the fetch kernel's load loop (bytes % 16 == 0).
cudaError_t launch_host_copy(void* dst, const void* src, size_t bytes, int blocks, cudaStream_t s);
// mcft_read_probe's kernels (csrc/probe.cu): pattern 0 contiguous, 1 the decode FFN's loads.
cudaError_t launch_read_probe(const void* buf, size_t bytes, int pattern, int row_bytes,
                              int blocks, unsigned* sink, cudaStream_t s);

// Fused decode prologue of one chained-stack layer at batch 1 (prologue.cu): residual update and
// RMSNorm, routing of layer l, cache step of layer l, prediction and prefetch event of layer l+1,
// permutation, in one launch of an 8-CTA cluster.
struct PrologueArgs {
  float* x;                // [1, d] fp32 stream (updated when y is given)
  const void* y;           // [1, d] previous layer's output (layer dtype) or NULL
  const void* gamma;       // [d] this layer's RMSNorm scale
  const void* gamma_next;  // [d] the next layer's (prediction), NULL: no prediction
  void* u;                 // [1, d] out: this layer's normalised input
  float eps;
  int d;
  RouteArgs route;         // this layer (route.x unused)
  RouteArgs pred;          // the next layer's prediction (when gamma_next is given)
  CacheStepArgs cache;     // this layer's step (cache.idx = route.idx)
  int do_prefetch;
  PrefetchArgs prefetch;   // the next layer's prefetch event (prefetch.idx = pred.idx)
  PermuteArgs perm;        // this layer's permutation (perm.idx = route.idx, T = 1)
};
bool prologue_supported(int d, int E, int T);
cudaError_t launch_prologue(const PrologueArgs& a, int dtype, cudaStream_t s);

// Residual update and RMSNorm of the stream entering a MoE block (norm.cu): x += y (when y is
// given), then u = gamma * x / sqrt(mean(x^2) + eps) (when gamma is given). One CTA per row.
struct NormArgs {
  float* x;            // [T, d] fp32 residual stream
  const void* y;       // [T, d] layer dtype or NULL
  const void* gamma;   // [d] layer dtype or NULL
  void* u;             // [T, d] layer dtype (written when gamma is given)
  int T, d;
  float eps;
};
cudaError_t launch_resid_norm(const NormArgs& a, int dtype, cudaStream_t s);

// Stage-1 mask machinery (mask.cu)
struct MaskSampleArgs {
  const float* m_tilde;   // [L, E]
  const float* uniforms;  // [L, E] in (0, 1)
  int L, E, e_keep;
  uint8_t* mask;          // [L, E] out
  float* pi;              // [L, E] out
  unsigned* err;
};
cudaError_t launch_mask_sample(const MaskSampleArgs& a, cudaStream_t s);

struct GateGradArgs {
  const void* dy;      // [T, d] layer dtype
  const float* o;      // forward workspace: expert output rows, ks planes o_plane apart
  const int* pos;      // forward workspace: permuted row of each assignment
  const WsHeader* hdr;
  size_t o_plane;
  int T, K, d, ks;
  float* dgate;        // [T, K] out
};
cudaError_t launch_gate_grad(const GateGradArgs& a, int dtype, cudaStream_t s);

struct MaskGradArgs {
  const int32_t* idx;   // [T, K]
  const float* gate;    // [T, K]
  const float* dgate;   // [T, K]
  const float* pi;      // [E]
  int T, K, E, gate_mode, accumulate;
  float* dm;            // [E] out: dL/dm
  float* dm_tilde;      // [E] out (or accumulated): dL/dm~
};
cudaError_t launch_mask_grad(const MaskGradArgs& a, cudaStream_t s);

unsigned* device_error_word();  // device address of the current device's error word
mcft_status set_error_message(mcft_status st, const char* msg);  // mcft_last_error() text

// The device-driven cached forward (mcft_moe_forward_cached); permuted = the workspace already
// holds this call's permutation (written by the fused prologue), so it is not recomputed.
mcft_status forward_cached_impl(const mcft_layer_desc* desc, const void* x, int T,
                                const int32_t* idx, const float* gate, mcft_cache* c, int layer,
                                const void* const* shared, void* y, void* workspace,
                                size_t ws_bytes, cudaStream_t compute_stream,
                                cudaStream_t copy_stream, bool permuted);

// One fused prologue launch for layer `layer` of a chained stack at batch 1 (prologue.cu): the
// stream update and norm, routing, the cache step, the next layer's prediction and prefetch event
// (when gamma_next is given and n_prefetch > 0), the permutation into `workspace`. Records the
// cache step's (and the prefetch's) events as mcft_cache_step / mcft_cache_prefetch do.
mcft_status stack_prologue(const mcft_layer_desc* desc, float* x, const void* y, const void* gamma,
                           const void* gamma_next, float eps, void* u, const void* w_router,
                           const float* prior, int32_t* idx, float* gate, const void* w_router_next,
                           const float* prior_next, int32_t* pred, float* gate_pred,
                           mcft_cache* c, int layer, int n_prefetch, void* workspace,
                           size_t ws_bytes, cudaStream_t stream);

// Kernel timing (profile.cu): event pairs around each launch while mcft_profile_enable(1) is on.
enum { kProfRoute, kProfCache, kProfPermute, kProfGather, kProfFfn13, kProfFfn2, kProfGemm13,
       kProfGemm2, kProfCombine, kProfDec13, kProfDec2, kProfFetch, kProfLora, kProfNorm,
       kProfPrefetch, kProfPfFetch, kProfPrologue, kProfDecFused, kProfHostCopy, kProfDecFetch,
       kProfGemm13Pair, kProfGemm2Pair, kProfCount };
void prof_begin(int kid, cudaStream_t s);
void prof_end(int kid, cudaStream_t s);

}  // namespace mcft
