// Per-layer expert cache decision kernel (Section 4.1 "Simulation", Eq. metrics).
//
// One warp per call: the lanes gather the distinct experts of the step (a 64-bit set) from the
// routing output, then apply the replacement rule (each slot choice a warp-wide reduction, the
// misses one at a time) on the layer's device-resident tag,
// last-use, insertion and access-count arrays: every expert of the step counts one access, hits
// refresh their last use, misses in ascending expert id take the lowest free slot or evict, among
// slots not used this step, the smallest key of the policy (LRU: last use, expert id; LFU: access
// count, last use, expert id; FIFO: insertion step, expert id), else go to a staging buffer for
// this step only (bypass). The miss list and the expert -> location map are written straight
// into host-mapped pinned memory, so the host can issue the fetches as soon as the step's event
// completes.
//
// Prefetch (offloading systems load experts ahead of need, Section 2; the rule is this library's):
// a prefetch is a cache event of its own, one time stamp between two steps. Its candidates are
// the experts of a predicted routing, ranked by how many predictions name them, then the best
// rank k at which a token predicts them, then the lower id. Every cached candidate is touched
// (last use = the event, no access counted); the n_max best-ranked uncached candidates, in
// ascending id, take the lowest free slot or evict, among slots not touched at the event, the
// smallest policy key. The
// loads form a separate fetch list, so a prefetch never disturbs the miss list of a step whose
// fetch may still be in flight. The next step counts hits on prefetched experts as useful, and
// leaves them out of its ready mask: their bytes arrive on the copy stream, so the FFN computes
// them with the step's misses, after the copies. Prefetched experts the step does not use are
// dropped first (slots freed) and flagged in the layer's cancel mask, which the prefetch's fetch
// kernel reads before each piece: a wrong prediction stops using the host link as soon as the
// step's routing is known.
#include "cache_warp.cuh"
#include "common.cuh"
#include "internal.h"

namespace mcft {
namespace {

__global__ void __launch_bounds__(32) cache_step_kernel(const __grid_constant__ CacheStepArgs a) {
  pdl_wait();
  cache_step_warp(a);
}

__global__ void __launch_bounds__(32) prefetch_kernel(const __grid_constant__ PrefetchArgs a) {
  pdl_wait();
  prefetch_warp(a);
}

// Copy the missed experts' blocks host -> device with 16-byte loads over the host link. Work
// units are 64 KB pieces of the missed blocks, spread over the grid.
__global__ void __launch_bounds__(256) fetch_kernel(const __grid_constant__ FetchArgs a) {
  pdl_wait();
  const int n = a.miss[0];
  const size_t words = a.bytes / 16, piece = kFetchPiece / 16;
  const size_t per = (words + piece - 1) / piece;
  const size_t units = size_t(n) * per;
  for (size_t u = blockIdx.x; u < units; u += gridDim.x) {
    const int e = a.miss[1 + int(u / per)];
    if (a.cancel) {  // a step dropped this prefetched expert: stop moving it (block-uniform read)
      __shared__ unsigned long long c;
      __syncthreads();
      if (threadIdx.x == 0) c = *reinterpret_cast<const volatile unsigned long long*>(a.cancel);
      __syncthreads();
      if ((c >> e) & 1ull) continue;
    }
    const uint4* src = reinterpret_cast<const uint4*>(a.host_src[e]);
    uint4* dst = reinterpret_cast<uint4*>(a.ptr_tab[e]);
    const size_t w0 = (u % per) * piece;
    const size_t w1 = w0 + piece < words ? w0 + piece : words;
    if (a.moved && threadIdx.x == 0) atomicAdd(a.moved, (unsigned long long)(w1 - w0) * 16ull);
    copy_piece(src, dst, w0, w1);
  }
}

// A plain copy of `words` 16-byte words from device-visible host memory with the fetch kernel's
// pieces and load loop: measures what SM loads get from the host link at a given grid size.
__global__ void __launch_bounds__(256) host_copy_kernel(const uint4* __restrict__ src,
                                                        uint4* __restrict__ dst, size_t words) {
  pdl_wait();
  const size_t piece = 4096;
  const size_t units = (words + piece - 1) / piece;
  for (size_t u = blockIdx.x; u < units; u += gridDim.x) {
    const size_t w0 = u * piece;
    copy_piece(src, dst, w0, w0 + piece < words ? w0 + piece : words);
  }
}

}  // namespace

cudaError_t launch_fetch(const FetchArgs& a, int blocks, cudaStream_t s, bool prefetch) {
  const int kid = prefetch ? kProfPfFetch : kProfFetch;
  prof_begin(kid, s);
  fetch_kernel<<<blocks, 256, 0, s>>>(a);
  prof_end(kid, s);
  return cudaGetLastError();
}

cudaError_t launch_host_copy(void* dst, const void* src, size_t bytes, int blocks, cudaStream_t s) {
  prof_begin(kProfHostCopy, s);
  host_copy_kernel<<<blocks, 256, 0, s>>>(static_cast<const uint4*>(src), static_cast<uint4*>(dst),
                                          bytes / 16);
  prof_end(kProfHostCopy, s);
  return cudaGetLastError();
}

cudaError_t launch_prefetch(const PrefetchArgs& a, cudaStream_t s) {
  prof_begin(kProfPrefetch, s);
  const cudaError_t e = launch_pdl(prefetch_kernel, dim3(1), dim3(32), 0, s, a);
  prof_end(kProfPrefetch, s);
  return e != cudaSuccess ? e : cudaGetLastError();
}

cudaError_t launch_cache_step(const CacheStepArgs& a, cudaStream_t s) {
  prof_begin(kProfCache, s);
  const cudaError_t e = launch_pdl(cache_step_kernel, dim3(1), dim3(32), 0, s, a);
  prof_end(kProfCache, s);
  return e != cudaSuccess ? e : cudaGetLastError();
}

}  // namespace mcft
