// Fused decode prologue of one layer of a chained stack at batch 1: everything a layer does
// before its expert FFN, in one launch of one thread-block cluster of 8 CTAs.
//
//   x <- x + y (the previous layer's output, when given);  u = RMSNorm_l(x)          (norm.cu rule)
//   z = W_l u; Top-K under the soft prior, gates                                     (Eq. inference)
//   cache step of layer l                                                            (Eq. metrics)
//   prediction of layer l+1: z' = W_{l+1} RMSNorm_{l+1}(x), its Top-K, and the prefetch event of
//   layer l+1 from it (when enabled)
//   permutation of the token's K assignments and the shared experts into segments
//
// The separate kernels (resid_norm, route twice, cache_step, prefetch, permute) each cost a launch
// and a few microseconds of latency at batch 1, and a single CTA reading a 256 KB router is slow.
// Here every CTA normalises the token (the first 256 threads follow the standalone norm kernel's
// element mapping and reduction order, so u is bit-identical), the cluster's 128 warps split both
// routers into (router, expert, contraction part) tasks, and each task's partial sum goes straight
// into the leader CTA's shared memory (distributed shared memory). After one cluster barrier the
// leader adds the parts in a fixed order, ranks both routings (the same warp function as the
// router kernel), then its warps run the cache step (layer l), the prefetch event (layer l+1) and
// the permutation concurrently (the same warp functions as the standalone kernels).
#include <cooperative_groups.h>

#include "cache_warp.cuh"
#include "common.cuh"
#include "internal.h"
#include "route_warp.cuh"

namespace mcft {
namespace {

namespace cg = cooperative_groups;

constexpr int kCluster = 8;
constexpr int kThreads = 512;
constexpr int kWarps = kThreads / 32;
constexpr int kMaxD = 4096;
constexpr int kMaxParts = 16;
constexpr int kNormThreads = 256;  // the standalone norm kernel's block size
constexpr int kRowVec = kMaxD / (4 * kNormThreads);  // float4 groups per norm thread
constexpr int kLoads = 8;  // 16-byte router loads a lane keeps in flight

template <typename TX>
struct Store;
template <>
struct Store<__nv_bfloat16> {
  using T = uint16_t;
  static constexpr int per16 = 8;
  __device__ static void put4(T* p, float4 v) {
    *reinterpret_cast<uint2*>(p) = make_uint2(pack2bf(v.x, v.y), pack2bf(v.z, v.w));
  }
  __device__ static float4 get4(const void* p) {
    const uint2 w = *reinterpret_cast<const uint2*>(p);
    return make_float4(bf16lo(w.x), bf16hi(w.x), bf16lo(w.y), bf16hi(w.y));
  }
  __device__ static void unpack(uint4 v, float* f) { unpack8(v, f); }
};
template <>
struct Store<float> {
  using T = float;
  static constexpr int per16 = 4;
  __device__ static void put4(T* p, float4 v) { *reinterpret_cast<float4*>(p) = v; }
  __device__ static float4 get4(const void* p) { return *reinterpret_cast<const float4*>(p); }
  __device__ static void unpack(uint4 v, float* f) {
    f[0] = __uint_as_float(v.x); f[1] = __uint_as_float(v.y);
    f[2] = __uint_as_float(v.z); f[3] = __uint_as_float(v.w);
  }
};

// Permutation of one token's K assignments (T = 1) and the S shared experts, one warp; writes
// what permute_kernel writes (segment sizes, offsets, row of each assignment, token of each row).
__device__ inline void permute_one_warp(const PermuteArgs& a) {
  __shared__ int offs[kMaxSeg + 1];
  const int lane = threadIdx.x & 31;
  const int n = a.K, nseg = a.E + a.S;
  const int e = lane < n ? a.idx[lane] : -1;
  const bool bad = __any_sync(0xffffffffu, lane < n && (e < 0 || e >= a.E));
  if (a.done)  // progress and claim counters: on every path, the abort path included
    for (int sg = lane; sg < nseg + kClaimSlots; sg += 32) a.done[sg] = 0;
  const unsigned peers = __match_any_sync(0xffffffffu, e);
  int vals[kMaxK];  // every lane sees the token's K expert ids
#pragma unroll
  for (int i = 0; i < kMaxK; ++i) vals[i] = __shfl_sync(0xffffffffu, e, i);
  if (bad) {
    if (lane == 0) {
      a.hdr->abort = 1;
      a.hdr->mrows = 0;
      set_error(a.err, kErrInvalid);
    }
    return;
  }
  int len[3], padded[3], sum = 0;
#pragma unroll
  for (int j = 0; j < 3; ++j) {
    const int sg = lane * 3 + j;
    len[j] = 0;
    if (sg < a.E) {
#pragma unroll
      for (int i = 0; i < kMaxK; ++i) len[j] += (i < n && vals[i] == sg) ? 1 : 0;
    } else if (sg < nseg) {
      len[j] = 1;  // a shared expert processes the token
    }
    padded[j] = (len[j] + a.pad - 1) / a.pad * a.pad;
    sum += padded[j];
  }
  int incl = sum;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int v = __shfl_up_sync(0xffffffffu, incl, o);
    if (lane >= o) incl += v;
  }
  int excl = incl - sum;
#pragma unroll
  for (int j = 0; j < 3; ++j) {
    const int sg = lane * 3 + j;
    if (sg < nseg) {
      offs[sg] = excl;
      a.off[sg] = excl;
      a.cnt[sg] = len[j];
      for (int r = 0; r < padded[j]; ++r) {
        const int row = excl + r;
        if (r >= len[j]) a.perm[row] = -1;
        else if (sg >= a.E) a.perm[row] = 0;
      }
    }
    excl += padded[j];
  }
  if (lane == 31) {
    offs[nseg] = incl;
    a.off[nseg] = incl;
    a.hdr->abort = 0;
    a.hdr->nseg = nseg;
    a.hdr->mrows = incl;
  }
  __syncwarp();
  if (lane < n) {  // stable within an expert: lower k first
    const int rank = __popc(peers & ((1u << lane) - 1u));
    const int row = offs[e] + rank;
    a.pos[lane] = row;
    a.perm[row] = 0;
  }
}

template <typename TX>
__global__ void __cluster_dims__(kCluster, 1, 1) __launch_bounds__(kThreads)
    prologue_kernel(const __grid_constant__ PrologueArgs a) {
  pdl_wait();
  using S = Store<TX>;
  using ST = typename S::T;
  __shared__ __align__(16) ST us[2][kMaxD];        // u, then the prediction's input
  __shared__ float part[2][kMaxE][kMaxParts];      // the leader's: partial logits
  __shared__ float zs[2][kMaxE];
  __shared__ float red[kNormThreads / 32];
  cg::cluster_group cluster = cg::this_cluster();
  const int crank = int(cluster.block_rank());
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int d = a.d, E = a.route.E;
  const int nr = a.gamma_next ? 2 : 1;

  // 1. the stream row and its norm(s), in registers of the first 256 threads; the scales are
  //    loaded with the row (one round trip for all of it)
  float4 v[kRowVec], gm[2][kRowVec];
  if (tid < kNormThreads) {
    float ss = 0.f;
#pragma unroll
    for (int i = 0; i < kRowVec; ++i) {
      const int c = tid * 4 + i * 4 * kNormThreads;
      if (c < d) {
        for (int q = 0; q < nr; ++q)
          gm[q][i] = S::get4(reinterpret_cast<const ST*>(q ? a.gamma_next : a.gamma) + c);
        v[i] = *reinterpret_cast<const float4*>(a.x + c);
        if (a.y) {
          const float4 y = S::get4(reinterpret_cast<const ST*>(a.y) + c);
          v[i].x += y.x; v[i].y += y.y; v[i].z += y.z; v[i].w += y.w;
        }
        ss = fmaf(v[i].x, v[i].x, ss);
        ss = fmaf(v[i].y, v[i].y, ss);
        ss = fmaf(v[i].z, v[i].z, ss);
        ss = fmaf(v[i].w, v[i].w, ss);
      }
    }
    ss = warp_sum(ss);
    if (lane == 0) red[warp] = ss;
  }
  __syncthreads();
  if (tid < kNormThreads) {
    float tot = 0.f;
#pragma unroll
    for (int w = 0; w < kNormThreads / 32; ++w) tot += red[w];
    const float r = 1.0f / sqrtf(tot / float(d) + a.eps);
#pragma unroll
    for (int i = 0; i < kRowVec; ++i) {
      const int c = tid * 4 + i * 4 * kNormThreads;
      if (c < d) {
        for (int q = 0; q < nr; ++q) {
          const float4 g = gm[q][i];
          S::put4(&us[q][c], make_float4(v[i].x * r * g.x, v[i].y * r * g.y, v[i].z * r * g.z,
                                        v[i].w * r * g.w));
        }
        if (crank == 0) S::put4(reinterpret_cast<ST*>(a.u) + c, S::get4(&us[0][c]));
      }
    }
  }
  __syncthreads();

  // 2. both routers as (router, expert, part) tasks over the cluster's warps
  const int nchunk = d / S::per16;
  // the split of a router does not depend on whether the prediction runs (budget of two routers),
  // so this layer's logits are bit-identical with and without prefetch
  int parts = 1;
  while (2 * parts <= kMaxParts && 2 * E * 2 * parts <= kCluster * kWarps && nchunk % (2 * parts) == 0)
    parts *= 2;
  const int per_part = nchunk / parts;
  const int tasks = nr * E * parts;
  float* lead = cluster.map_shared_rank(&part[0][0][0], 0);
  for (int task = crank * kWarps + warp; task < tasks; task += kCluster * kWarps) {
    const int q = task / (E * parts), rem = task % (E * parts);
    const int e = rem / parts, pt = rem % parts;
    const RouteArgs& ra = q ? a.pred : a.route;
    const char* wrow = reinterpret_cast<const char*>(ra.w_router) + (size_t(e) * nchunk + size_t(pt) * per_part) * 16;
    const char* urow = reinterpret_cast<const char*>(&us[q][0]) + size_t(pt) * per_part * 16;
    float acc = 0.f;
    for (int base = 0; base < per_part; base += 32 * kLoads) {  // kLoads row loads in flight
      uint4 wv[kLoads];
#pragma unroll
      for (int i = 0; i < kLoads; ++i) {
        const int c = base + i * 32 + lane;
        if (c < per_part) wv[i] = ldg16(wrow + size_t(c) * 16);
      }
#pragma unroll
      for (int i = 0; i < kLoads; ++i) {
        const int c = base + i * 32 + lane;
        if (c < per_part) {
          float wf[S::per16], uf[S::per16];
          S::unpack(wv[i], wf);
          S::unpack(*reinterpret_cast<const uint4*>(urow + size_t(c) * 16), uf);
#pragma unroll
          for (int j = 0; j < S::per16; ++j) acc = fmaf(uf[j], wf[j], acc);
        }
      }
    }
    acc = warp_sum(acc);
    if (lane == 0) lead[(q * kMaxE + e) * kMaxParts + pt] = acc;
  }
  cluster.sync();  // every partial logit is in the leader's shared memory
  if (crank != 0) return;

  // 3. the leader: logits, ranking, then cache step / prefetch / permutation on separate warps
  if (a.y && tid < kNormThreads) {  // the updated stream (every CTA has read x by now)
#pragma unroll
    for (int i = 0; i < kRowVec; ++i) {
      const int c = tid * 4 + i * 4 * kNormThreads;
      if (c < d) *reinterpret_cast<float4*>(a.x + c) = v[i];
    }
  }
  for (int i = tid; i < nr * E; i += kThreads) {
    const int q = i / E, e = i % E;
    float z = 0.f;
    for (int p = 0; p < parts; ++p) z += part[q][e][p];
    zs[q][e] = z;
  }
  __syncthreads();
  if (warp == 0) rank_and_gate_warp(a.route, zs[0], 0);
  else if (warp == 1 && nr == 2) rank_and_gate_warp(a.pred, zs[1], 0);
  __syncthreads();  // idx and the prediction are in global memory, visible to the whole CTA
  if (warp == 0) cache_step_warp(a.cache);
  else if (warp == 1 && nr == 2 && a.do_prefetch) prefetch_warp(a.prefetch);
  else if (warp == 2) permute_one_warp(a.perm);
}

}  // namespace

bool prologue_supported(int d, int E, int T) { return T == 1 && d <= kMaxD && E <= kMaxE; }

cudaError_t launch_prologue(const PrologueArgs& a, int dtype, cudaStream_t s) {
  prof_begin(kProfPrologue, s);
  const cudaError_t e = dtype == MCFT_BF16
      ? launch_pdl(prologue_kernel<__nv_bfloat16>, dim3(kCluster), dim3(kThreads), 0, s, a)
      : launch_pdl(prologue_kernel<float>, dim3(kCluster), dim3(kThreads), 0, s, a);
  prof_end(kProfPrologue, s);
  return e != cudaSuccess ? e : cudaGetLastError();
}

}  // namespace mcft
