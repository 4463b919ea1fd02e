// Token permutation by expert: histogram, exclusive scan of padded segment sizes, and a stable
// scatter (assignments keep their (t, k) order inside each expert), plus the row gather that builds
// the permuted activation matrix for the tensor-core path. Segments E..E+S-1 hold the shared
// experts, which process every token (Section 3.1).
#include "common.cuh"
#include "internal.h"

namespace mcft {
namespace {

constexpr int kThreads = 1024;

__global__ void __launch_bounds__(kThreads) permute_kernel(const __grid_constant__ PermuteArgs a) {
  pdl_wait();
  __shared__ int hist[kMaxSeg];
  __shared__ int run[kMaxE];
  __shared__ int offs[kMaxSeg + 1];
  __shared__ int wcnt[kThreads / 32][kMaxE];
  __shared__ int bad;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int n = a.T * a.K, nseg = a.E + a.S;
  if (tid < kMaxSeg) hist[tid] = 0;
  if (tid < kMaxE) run[tid] = 0;
  if (tid == 0) bad = 0;
  __syncthreads();
  for (int i = tid; i < n; i += kThreads) {
    const int e = a.idx[i];
    if (e < 0 || e >= a.E) bad = 1;
    else atomicAdd(&hist[e], 1);
  }
  __syncthreads();
  // progress and claim counters: on every path, the abort path included
  if (a.done && tid < nseg + kClaimSlots) a.done[tid] = 0;
  if (bad) {
    if (tid == 0) {
      a.hdr->abort = 1;
      a.hdr->mrows = 0;
      set_error(a.err, kErrInvalid);
    }
    return;
  }
  // padded exclusive scan of the segment sizes: warp 0, three segments per lane (kMaxSeg <= 96)
  if (warp == 0) {
    int len[3], padded[3], sum = 0;
#pragma unroll
    for (int j = 0; j < 3; ++j) {
      const int sg = lane * 3 + j;
      len[j] = sg < nseg ? (sg < a.E ? hist[sg] : a.T) : 0;
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
  }
  __syncthreads();

  const unsigned lt_mask = (1u << lane) - 1u;
  for (int base = 0; base < n; base += kThreads) {
    const int i = base + tid;
    const bool valid = i < n;
    const int e = valid ? a.idx[i] : -1;
    for (int j = tid; j < (kThreads / 32) * kMaxE; j += kThreads) (&wcnt[0][0])[j] = 0;
    __syncthreads();
    const unsigned peers = __match_any_sync(0xffffffffu, e);
    const int rank = __popc(peers & lt_mask);
    if (valid && rank == 0) wcnt[warp][e] = __popc(peers);
    __syncthreads();
    if (valid) {
      int p = run[e] + rank;
      for (int w = 0; w < warp; ++w) p += wcnt[w][e];
      const int row = offs[e] + p;
      a.pos[i] = row;
      a.perm[row] = i / a.K;
    }
    __syncthreads();
    if (tid < a.E) {
      int tot = 0;
      for (int w = 0; w < kThreads / 32; ++w) tot += wcnt[w][tid];
      run[tid] += tot;
    }
    __syncthreads();
  }
  // padding rows of routed segments; shared segments list every token in order. One thread per
  // row; its segment is found by binary search on the offsets.
  const int mrows = offs[nseg];
  for (int r = tid; r < mrows; r += kThreads) {
    int lo = 0, hi = nseg;  // largest segment with offs[seg] <= r
    while (hi - lo > 1) {
      const int mid = (lo + hi) >> 1;
      if (offs[mid] <= r) lo = mid;
      else hi = mid;
    }
    const int len = lo < a.E ? hist[lo] : a.T;
    const int local = r - offs[lo];
    if (lo >= a.E && local < len) a.perm[r] = local;
    else if (local >= len) a.perm[r] = -1;
  }
}

// xp[r, :] = x[perm[r], :] (bf16), zero rows for padding.
__global__ void __launch_bounds__(256) gather_kernel(const __grid_constant__ GatherArgs a) {
  pdl_wait();
  if (a.hdr->abort) return;
  const int mrows = a.hdr->mrows;
  const int nch = a.d / 8;  // 16-byte chunks per row
  for (int r = blockIdx.x; r < mrows; r += gridDim.x) {
    const int t = a.perm[r];
    uint4* dst = reinterpret_cast<uint4*>(reinterpret_cast<char*>(a.xp) + size_t(r) * a.d * 2);
    if (t < 0) {
      for (int c = threadIdx.x; c < nch; c += blockDim.x) dst[c] = make_uint4(0, 0, 0, 0);
    } else {
      const uint4* src =
          reinterpret_cast<const uint4*>(reinterpret_cast<const char*>(a.x) + size_t(t) * a.d * 2);
      for (int c = threadIdx.x; c < nch; c += blockDim.x) dst[c] = ldg16(src + c);
    }
  }
}

}  // namespace

cudaError_t launch_permute(const PermuteArgs& a, cudaStream_t s) {
  prof_begin(kProfPermute, s);
  const cudaError_t e = launch_pdl(permute_kernel, dim3(1), dim3(kThreads), 0, s, a);
  prof_end(kProfPermute, s);
  return e != cudaSuccess ? e : cudaGetLastError();
}

cudaError_t launch_gather(const GatherArgs& a, cudaStream_t s) {
  const int grid = a.mcap < 4096 ? (a.mcap > 0 ? a.mcap : 1) : 4096;
  prof_begin(kProfGather, s);
  const cudaError_t e = launch_pdl(gather_kernel, dim3(grid), dim3(256), 0, s, a);
  prof_end(kProfGather, s);
  return e != cudaSuccess ? e : cudaGetLastError();
}

}  // namespace mcft
