// Per-layer expert cache decision kernel (Section 4.1 "Simulation", Eq. metrics).
//
// One warp per call: the lanes gather the distinct experts of the step (a 64-bit set) from the
// routing output, then lane 0 applies the replacement rule on the layer's device-resident tag,
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
#include "common.cuh"
#include "internal.h"

namespace mcft {
namespace {

// True when slot s precedes slot v in eviction order under the policy's key.
__device__ __forceinline__ bool victim_before(int policy, int s, int v, const int32_t* tag,
                                              const int64_t* last, const int64_t* ins,
                                              const int64_t* freq) {
  if (policy == MCFT_CACHE_LFU) {
    const int64_t fs = freq[tag[s]], fv = freq[tag[v]];
    if (fs != fv) return fs < fv;
  } else if (policy == MCFT_CACHE_FIFO) {
    if (ins[s] != ins[v]) return ins[s] < ins[v];
    return tag[s] < tag[v];
  }
  if (last[s] != last[v]) return last[s] < last[v];
  return tag[s] < tag[v];
}

__global__ void __launch_bounds__(32) cache_step_kernel(const __grid_constant__ CacheStepArgs a) {
  pdl_wait();
  __shared__ int32_t s_tag[kMaxE];
  __shared__ int64_t s_last[kMaxE], s_ins[kMaxE], s_freq[kMaxE];
  __shared__ int32_t s_out[1 + 3 * kMaxE];  // n_miss, miss experts, miss locations, loc_of
  const int lane = threadIdx.x;
  const int B = a.B, E = a.E;
  unsigned long long mine = 0;
  int bad = 0;
  for (int i = lane; i < a.n; i += 32) {
    const int e = a.idx[i];
    if (e < 0 || e >= E) bad = 1;
    else mine |= 1ull << e;
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    mine |= __shfl_xor_sync(0xffffffffu, mine, o);
    bad |= __shfl_xor_sync(0xffffffffu, bad, o);
  }
  if (bad) {  // no state change on bad input
    if (lane == 0) {
      set_error(a.err, kErrInvalid);
      a.miss_out[0] = 0;
      a.miss_dev[0] = 0;
      *a.ready = 0;
    }
    for (int e = lane; e < E; e += 32) a.ptr_tab[e] = 0;
    __threadfence_system();
    return;
  }
  int32_t* tag = a.tag + size_t(a.layer) * B;
  int64_t* last = a.last + size_t(a.layer) * B;
  int64_t* ins = a.ins + size_t(a.layer) * B;
  int64_t* freq = a.freq + size_t(a.layer) * E;
  // stage the layer's state in shared memory (one load per lane)
  for (int i = lane; i < B; i += 32) {
    s_tag[i] = tag[i];
    s_last[i] = last[i];
    s_ins[i] = ins[i];
  }
  for (int e = lane; e < E; e += 32) s_freq[e] = freq[e] + ((mine >> e) & 1ull);
  __syncwarp();
  unsigned long long cached = 0, pf = 0;
  int hits = 0, nm = 0, nbyp = 0;
  const int64_t t = a.step[a.layer];
  if (lane == 0) {
    int32_t* m_exp = s_out + 1;
    int32_t* m_loc = s_out + 1 + E;
    int32_t* loc_of = s_out + 1 + 2 * E;
    for (int e = 0; e < E; ++e) loc_of[e] = -1;
    pf = a.pfmask[a.layer];
    const unsigned long long drop = pf & ~mine;  // prefetched experts this step does not use
    for (int sl = 0; sl < B; ++sl) {
      const int e = s_tag[sl];
      if (e >= 0 && ((drop >> e) & 1ull)) {
        s_tag[sl] = -1;
        s_last[sl] = -1;
        s_ins[sl] = -1;
      }
    }
    a.cancel[a.layer] = drop;
    for (int sl = 0; sl < B; ++sl) {
      const int e = s_tag[sl];
      if (e < 0) continue;
      cached |= 1ull << e;
      if ((mine >> e) & 1ull) {
        s_last[sl] = t;
        loc_of[e] = sl;
        ++hits;
      }
    }
    const int useful = __popcll(pf & mine & cached);
    unsigned long long miss = mine & ~cached;
    while (miss) {
      const int e = __ffsll(static_cast<long long>(miss)) - 1;  // ascending expert id
      miss &= miss - 1;
      int slot = -1;
      for (int sl = 0; sl < B; ++sl)
        if (s_tag[sl] < 0) { slot = sl; break; }
      if (slot < 0) {
        for (int sl = 0; sl < B; ++sl) {
          if (s_last[sl] >= t) continue;  // used at this step: never a victim
          if (slot < 0 || victim_before(a.policy, sl, slot, s_tag, s_last, s_ins, s_freq)) slot = sl;
        }
      }
      m_exp[nm] = e;
      if (slot < 0) {
        m_loc[nm] = -1;
        loc_of[e] = B + nbyp;
        ++nbyp;
      } else {
        s_tag[slot] = e;
        s_last[slot] = t;
        s_ins[slot] = t;
        m_loc[nm] = slot;
        loc_of[e] = slot;
      }
      ++nm;
    }
    s_out[0] = nm;
    a.step[a.layer] = t + 1;
    unsigned long long* c = a.counters + size_t(a.layer) * kCacheCounters;
    c[0] += hits;
    c[1] += nm;
    c[2] += nbyp;
    c[4] += useful;
    a.pfmask[a.layer] = 0;
  }
  cached = __shfl_sync(0xffffffffu, cached, 0);
  pf = __shfl_sync(0xffffffffu, pf, 0);
  __syncwarp();
  // write back the state and publish the step's miss list and expert table (all lanes)
  for (int i = lane; i < B; i += 32) {
    tag[i] = s_tag[i];
    last[i] = s_last[i];
    ins[i] = s_ins[i];
  }
  for (int e = lane; e < E; e += 32) freq[e] = s_freq[e];
  for (int i = lane; i < 1 + 3 * E; i += 32) {
    a.miss_out[i] = s_out[i];
    a.miss_dev[i] = s_out[i];
  }
  unsigned long long hitbits = 0;
  for (int e = lane; e < E; e += 32) {
    const int loc = s_out[1 + 2 * E + e];
    unsigned long long p = 0;
    if (loc >= 0 && a.slots)
      p = reinterpret_cast<unsigned long long>(loc < B ? a.slots + size_t(loc) * a.expert_bytes
                                                       : a.staging + size_t(loc - B) * a.expert_bytes);
    a.ptr_tab[e] = p;
    // ready now: hits whose bytes are not still coming from a prefetch
    if (loc >= 0 && loc < B && ((cached & ~pf) >> e) & 1ull) hitbits |= 1ull << e;
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) hitbits |= __shfl_xor_sync(0xffffffffu, hitbits, o);
  if (lane == 0) *a.ready = hitbits;
  __threadfence_system();
}

// Prefetch decision (one warp). The lanes count how many predicted (token, k) entries name each
// expert; lane 0 ranks, touches, claims slots and writes the fetch list.
__global__ void __launch_bounds__(32) prefetch_kernel(const __grid_constant__ PrefetchArgs a) {
  pdl_wait();
  __shared__ int cnt[kMaxE], rank[kMaxE];
  __shared__ int32_t s_tag[kMaxE];
  __shared__ int64_t s_last[kMaxE], s_ins[kMaxE], s_freq[kMaxE];
  __shared__ int32_t s_list[1 + kMaxE];
  const int lane = threadIdx.x, B = a.B, E = a.E;
  for (int e = lane; e < E; e += 32) {
    cnt[e] = 0;
    rank[e] = 1 << 30;
  }
  __syncwarp();
  int bad = 0;
  for (int i = lane; i < a.n; i += 32) {
    const int e = a.idx[i];
    if (e < 0 || e >= E) {
      bad = 1;
    } else {
      atomicAdd(&cnt[e], 1);
      atomicMin(&rank[e], i % a.K);
    }
  }
  bad = __any_sync(0xffffffffu, bad);
  if (bad) {  // no state change on bad input
    if (lane == 0) {
      set_error(a.err, kErrInvalid);
      a.list[0] = 0;
    }
    return;
  }
  int32_t* tag = a.tag + size_t(a.layer) * B;
  int64_t* last = a.last + size_t(a.layer) * B;
  int64_t* ins = a.ins + size_t(a.layer) * B;
  for (int i = lane; i < B; i += 32) {
    s_tag[i] = tag[i];
    s_last[i] = last[i];
    s_ins[i] = ins[i];
  }
  for (int e = lane; e < E; e += 32) s_freq[e] = a.freq[size_t(a.layer) * E + e];
  __syncwarp();
  if (lane == 0) {
    const int64_t t = a.step[a.layer];
    // every cached candidate is touched; the loads are the n_max best-ranked uncached candidates
    // by (count descending, best rank ascending, id ascending)
    unsigned long long cand = 0, cached = 0;
    for (int e = 0; e < E; ++e)
      if (cnt[e] > 0) cand |= 1ull << e;
    for (int sl = 0; sl < B; ++sl) {
      const int e = s_tag[sl];
      if (e < 0) continue;
      cached |= 1ull << e;
      if ((cand >> e) & 1ull) s_last[sl] = t;
    }
    unsigned long long load = 0;
    for (int j = 0; j < a.n_max; ++j) {
      int best = -1;
      for (int e = 0; e < E; ++e) {
        if (!(((cand & ~cached & ~load) >> e) & 1ull)) continue;
        if (best < 0 || cnt[e] > cnt[best] || (cnt[e] == cnt[best] && rank[e] < rank[best])) best = e;
      }
      if (best < 0) break;
      load |= 1ull << best;
    }
    unsigned long long pf = a.pfmask[a.layer];
    int nl = 0;
    while (load) {
      const int e = __ffsll(static_cast<long long>(load)) - 1;
      load &= load - 1;
      int slot = -1;
      for (int sl = 0; sl < B; ++sl)
        if (s_tag[sl] < 0) { slot = sl; break; }
      if (slot < 0) {
        for (int sl = 0; sl < B; ++sl) {
          if (s_last[sl] >= t) continue;  // touched at this event: never a victim
          if (slot < 0 || victim_before(a.policy, sl, slot, s_tag, s_last, s_ins, s_freq)) slot = sl;
        }
      }
      if (slot < 0) continue;  // unreachable with n_max <= B; kept for safety
      if (s_tag[slot] >= 0) pf &= ~(1ull << s_tag[slot]);
      s_tag[slot] = e;
      s_last[slot] = t;
      s_ins[slot] = t;
      pf |= 1ull << e;
      s_list[1 + nl] = e;
      ++nl;
    }
    s_list[0] = nl;
    a.pfmask[a.layer] = pf;
    a.cancel[a.layer] = 0;
    a.step[a.layer] = t + 1;
    a.counters[size_t(a.layer) * kCacheCounters + 3] += nl;
  }
  __syncwarp();
  for (int i = lane; i < B; i += 32) {
    tag[i] = s_tag[i];
    last[i] = s_last[i];
    ins[i] = s_ins[i];
  }
  const int nl = s_list[0];
  for (int i = lane; i <= nl; i += 32) a.list[i] = s_list[i];
  for (int e = lane; e < E; e += 32) a.ptr_tab[e] = 0;
  __syncwarp();
  for (int i = lane; i < nl; i += 32) {
    const int e = s_list[1 + i];
    int slot = 0;
    for (int sl = 0; sl < B; ++sl)
      if (s_tag[sl] == e) slot = sl;
    a.ptr_tab[e] = a.slots ? reinterpret_cast<unsigned long long>(a.slots + size_t(slot) * a.expert_bytes)
                           : 0ull;
  }
}

// Copy the missed experts' blocks host -> device with 16-byte loads over the host link. Work
// units are 64 KB pieces of the missed blocks, spread over the grid.
__global__ void __launch_bounds__(256) fetch_kernel(const __grid_constant__ FetchArgs a) {
  pdl_wait();
  const int n = a.miss[0];
  const size_t words = a.bytes / 16, piece = 4096;
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
    const size_t stride = blockDim.x;
    for (size_t w = w0 + threadIdx.x; w < w1; w += 4 * stride) {
      uint4 v[4];
#pragma unroll
      for (int j = 0; j < 4; ++j)
        if (w + j * stride < w1) v[j] = src[w + j * stride];
#pragma unroll
      for (int j = 0; j < 4; ++j)
        if (w + j * stride < w1) dst[w + j * stride] = v[j];
    }
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
