// Internal launchers and the workspace layout shared by the C ABI (api.cu) and the kernels.
#pragma once

#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

#include "../../include/mcft.h"

namespace mcft {

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

// Header at the start of the forward workspace.
struct WsHeader {
  int abort;     // set when a kernel of this call found bad data; later kernels skip their work
  int nseg;      // E + n_shared
  int mrows;     // total permuted rows (padded)
  int pad0;
};

// Device workspace of one mcft_moe_forward call. Segments 0..E-1 are the routed experts,
// E..E+S-1 the shared experts (every token). Offsets are in permuted rows.
struct WsLayout {
  bool tc;        // tensor-core path (bf16, large T)
  bool decode;    // bf16 decode path (T <= 64)
  int pad;        // rows per segment are padded to a multiple of this (128 on the TC path)
  int mcap;       // capacity in permuted rows
  int ks;         // partial planes of o (contraction split of the decode GEMM2)
  size_t hdr, cnt, off, pos, perm, xp, h, o, total;
};
WsLayout ws_layout(int d, int E, int K, int w, int S, int dtype, int T);

struct PermuteArgs {
  const int32_t* idx;
  int T, K, E, S, pad, mcap;
  WsHeader* hdr;
  int* cnt;    // [E+S] rows per segment (unpadded)
  int* off;    // [E+S+1] padded segment offsets
  int* pos;    // [T*K] permuted row of assignment (t, k)
  int* perm;   // [mcap] token of each permuted row, -1 for padding
  unsigned* err;
};
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
};

// Segment s of a forward: its block address and whether this launch computes it.
__device__ __forceinline__ const void* seg_block(const FfnArgs& a, int s) {
  return (a.wtab && s < a.E) ? reinterpret_cast<const void*>(a.wtab[s]) : a.wblk[s];
}
__device__ __forceinline__ bool seg_in_phase(const FfnArgs& a, int s, unsigned long long hits) {
  if (a.phase == 0) return true;
  const bool hit = s >= a.E || ((hits >> s) & 1ull);
  return a.phase == 1 ? hit : !hit;
}
cudaError_t launch_ffn_rowwise(const FfnArgs& a, int dtype, int num_sms, cudaStream_t s);  // fp32
cudaError_t launch_ffn_decode(const FfnArgs& a, int num_sms, cudaStream_t s);  // bf16, T <= 64
int decode_ksplit(int T);  // contraction split of the decode GEMM2 for T tokens
cudaError_t launch_ffn_tc(const FfnArgs& a, const void* xp, int mcap, int num_sms, cudaStream_t s);

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
  unsigned long long* counters;  // [L*3] hits, fetches, bypass
  int32_t* miss_out;  // host-mapped, per layer: [n_miss, expert[E], loc[E], loc_of[E]]
  int32_t* miss_dev;  // device copy of the same list (read by the fetch kernel)
  unsigned long long* ptr_tab;  // device [E]: block address of each selected expert, else 0
  unsigned long long* ready;    // device: bit e set when expert e was a hit at this step
  const char* slots;            // this layer's first slot block (NULL in accounting mode)
  const char* staging;          // bypass staging blocks
  size_t expert_bytes;
  unsigned* err;
};
cudaError_t launch_cache_step(const CacheStepArgs& a, cudaStream_t s);

// Device-driven fetch: copy the blocks of a layer's missed experts from pinned host memory
// (device-visible addresses host_src[E]) into the addresses ptr_tab[E] chosen by the cache step.
struct FetchArgs {
  const int32_t* miss;                // device miss list of the layer [1 + 3E]
  const unsigned long long* host_src; // [E]
  const unsigned long long* ptr_tab;  // [E]
  size_t bytes;                       // per expert block, multiple of 16
};
cudaError_t launch_fetch(const FetchArgs& a, int blocks, cudaStream_t s);

unsigned* device_error_word();  // device address of the current device's error word
mcft_status set_error_message(mcft_status st, const char* msg);  // mcft_last_error() text

// Kernel timing (profile.cu): event pairs around each launch while mcft_profile_enable(1) is on.
enum { kProfRoute, kProfCache, kProfPermute, kProfGather, kProfFfn13, kProfFfn2, kProfGemm13,
       kProfGemm2, kProfCombine, kProfDec13, kProfDec2, kProfFetch, kProfCount };
void prof_begin(int kid, cudaStream_t s);
void prof_end(int kid, cudaStream_t s);

}  // namespace mcft
