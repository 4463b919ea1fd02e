// Token permutation by expert: histogram, exclusive scan of padded segment sizes, and a stable
// scatter (assignments keep their (t, k) order inside each expert), plus the row gather that builds
// the permuted activation matrix for the tensor-core path. Segments E..E+S-1 hold the shared
// experts, which process every token (Section 3.1). The stable order defines the result uniquely,
// so the one-CTA kernel (decode batches) and the three chunked launches (large batches) write the
// same rows.
#include "common.cuh"
#include "internal.h"

namespace mcft {
namespace {

constexpr int kThreads = 1024;

// Padded exclusive scan of the segment sizes by warp 0 (three segments per lane, kMaxSeg <= 96):
// writes offs (shared), a.off, a.cnt and the header.
__device__ void scan_segments(const PermuteArgs& a, const int* hist, int* offs, int lane) {
  const int nseg = a.E + a.S;
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

// Stable scatter of assignments [i0, i1) (all threads of the CTA, kThreads of them): each
// assignment's row is offs[e] + run[e] + (earlier assignments of e in this round); run[e] holds the
// number of earlier assignments of e before the round and is advanced by it.
__device__ void scatter_rounds(const PermuteArgs& a, int i0, int i1, const int* offs, int* run,
                               int (*wcnt)[kMaxE]) {
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const unsigned lt_mask = (1u << lane) - 1u;
  for (int base = i0; base < i1; base += kThreads) {
    const int i = base + tid;
    const bool valid = i < i1;
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
}

// Padding rows of routed segments (-1) and the rows of shared segments (every token in order):
// rows r0, r0 + stride, ... of [0, mrows); a row's segment is found by binary search on offs.
__device__ void fill_rows(const PermuteArgs& a, const int* offs, const int* len_of, int r0,
                          int stride) {
  const int nseg = a.E + a.S;
  const int mrows = offs[nseg];
  for (int r = r0; r < mrows; r += stride) {
    int lo = 0, hi = nseg;  // largest segment with offs[seg] <= r
    while (hi - lo > 1) {
      const int mid = (lo + hi) >> 1;
      if (offs[mid] <= r) lo = mid;
      else hi = mid;
    }
    const int len = lo < a.E ? len_of[lo] : a.T;
    const int local = r - offs[lo];
    if (lo >= a.E && local < len) a.perm[r] = local;
    else if (local >= len) a.perm[r] = -1;
  }
}

// One CTA for the whole call (decode batches: a few microseconds).
__global__ void __launch_bounds__(kThreads) permute_kernel(const __grid_constant__ PermuteArgs a) {
  pdl_wait();
  // the next launch (the decode FFN) may start now: before its own wait it reads only what was
  // written before this kernel started (its parameters, the cache's expert table)
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
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
  if (warp == 0) scan_segments(a, hist, offs, lane);
  __syncthreads();
  scatter_rounds(a, 0, n, offs, run, wcnt);
  fill_rows(a, offs, hist, tid, kThreads);
}

// Large batches (prefill, fine-tuning): the same permutation by three launches over chunks of
// kChunk assignments. The scratch holds, per chunk, its per-expert counts (turned into the
// chunk's first position inside each expert) and whether it saw an invalid id.
constexpr int kChunk = 1024;

__device__ __forceinline__ int* chunk_row(const PermuteArgs& a, int c) { return a.scr + c * kMaxE; }
__device__ __forceinline__ int* chunk_bad(const PermuteArgs& a) { return a.scr + kPermChunks * kMaxE; }

__global__ void __launch_bounds__(256) permute_count_kernel(const __grid_constant__ PermuteArgs a,
                                                            int chunk) {
  pdl_wait();
  __shared__ int hist[kMaxE];
  __shared__ int bad;
  const int tid = threadIdx.x, c = blockIdx.x;
  if (tid < kMaxE) hist[tid] = 0;
  if (tid == 0) bad = 0;
  __syncthreads();
  const int n = a.T * a.K, i1 = min(n, (c + 1) * chunk);
  for (int i = c * chunk + tid; i < i1; i += blockDim.x) {
    const int e = a.idx[i];
    if (e < 0 || e >= a.E) bad = 1;
    else atomicAdd(&hist[e], 1);
  }
  __syncthreads();
  if (tid < a.E) chunk_row(a, c)[tid] = hist[tid];
  if (tid == 0) chunk_bad(a)[c] = bad;
}

__global__ void __launch_bounds__(kThreads) permute_scan_kernel(const __grid_constant__ PermuteArgs a,
                                                                int nchunks) {
  pdl_wait();
  __shared__ int hist[kMaxSeg];
  __shared__ int offs[kMaxSeg + 1];
  __shared__ int bad;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int nseg = a.E + a.S;
  if (tid == 0) {
    int b = 0;
    for (int c = 0; c < nchunks; ++c) b |= chunk_bad(a)[c];
    bad = b;
  }
  if (tid < a.E) {  // expert tid: its total, and each chunk's first position inside the expert
    int run = 0;
    for (int c = 0; c < nchunks; ++c) {
      int* r = chunk_row(a, c);
      const int v = r[tid];
      r[tid] = run;
      run += v;
    }
    hist[tid] = run;
  }
  __syncthreads();
  if (a.done && tid < nseg + kClaimSlots) a.done[tid] = 0;
  if (bad) {
    if (tid == 0) {
      a.hdr->abort = 1;
      a.hdr->mrows = 0;
      set_error(a.err, kErrInvalid);
    }
    return;
  }
  if (warp == 0) scan_segments(a, hist, offs, lane);
}

__global__ void __launch_bounds__(kThreads) permute_scatter_kernel(const __grid_constant__ PermuteArgs a,
                                                                   int chunk) {
  pdl_wait();
  __shared__ int len[kMaxSeg];
  __shared__ int run[kMaxE];
  __shared__ int offs[kMaxSeg + 1];
  __shared__ int wcnt[kThreads / 32][kMaxE];
  const int tid = threadIdx.x, c = blockIdx.x;
  if (a.hdr->abort) return;
  const int n = a.T * a.K, nseg = a.E + a.S;
  if (tid <= nseg) offs[tid] = a.off[tid];
  if (tid < nseg) len[tid] = a.cnt[tid];
  if (tid < a.E) run[tid] = chunk_row(a, c)[tid];
  __syncthreads();
  scatter_rounds(a, c * chunk, min(n, (c + 1) * chunk), offs, run, wcnt);
  fill_rows(a, offs, len, c * kThreads + tid, gridDim.x * kThreads);
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
  const int n = a.T * a.K;
  prof_begin(kProfPermute, s);
  cudaError_t e;
  if (a.scr == nullptr || n <= kPermSingleMax) {
    e = launch_pdl(permute_kernel, dim3(1), dim3(kThreads), 0, s, a);
  } else {
    int nchunks = (n + kChunk - 1) / kChunk;
    if (nchunks > kPermChunks) nchunks = kPermChunks;
    const int chunk = (n + nchunks - 1) / nchunks;
    e = launch_pdl(permute_count_kernel, dim3(nchunks), dim3(256), 0, s, a, chunk);
    if (e == cudaSuccess) e = launch_pdl(permute_scan_kernel, dim3(1), dim3(kThreads), 0, s, a, nchunks);
    if (e == cudaSuccess) e = launch_pdl(permute_scatter_kernel, dim3(nchunks), dim3(kThreads), 0, s, a, chunk);
  }
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
