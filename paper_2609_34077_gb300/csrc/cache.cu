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
  unsigned long long cached = 0;
  int hits = 0, nm = 0, nbyp = 0;
  const int64_t t = a.step[a.layer];
  if (lane == 0) {
    int32_t* m_exp = s_out + 1;
    int32_t* m_loc = s_out + 1 + E;
    int32_t* loc_of = s_out + 1 + 2 * E;
    for (int e = 0; e < E; ++e) loc_of[e] = -1;
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
    unsigned long long* c = a.counters + size_t(a.layer) * 3;
    c[0] += hits;
    c[1] += nm;
    c[2] += nbyp;
  }
  cached = __shfl_sync(0xffffffffu, cached, 0);
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
    if (loc >= 0 && loc < B && ((cached >> e) & 1ull)) hitbits |= 1ull << e;
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) hitbits |= __shfl_xor_sync(0xffffffffu, hitbits, o);
  if (lane == 0) *a.ready = hitbits;
  __threadfence_system();
}

// Copy the missed experts' blocks host -> device with 16-byte loads over the host link. Work
// units are 64 KB pieces of the missed blocks, spread over the grid.
__global__ void __launch_bounds__(256) fetch_kernel(const __grid_constant__ FetchArgs a) {
  const int n = a.miss[0];
  const size_t words = a.bytes / 16, piece = 4096;
  const size_t per = (words + piece - 1) / piece;
  const size_t units = size_t(n) * per;
  for (size_t u = blockIdx.x; u < units; u += gridDim.x) {
    const int e = a.miss[1 + int(u / per)];
    const uint4* src = reinterpret_cast<const uint4*>(a.host_src[e]);
    uint4* dst = reinterpret_cast<uint4*>(a.ptr_tab[e]);
    const size_t w0 = (u % per) * piece;
    const size_t w1 = w0 + piece < words ? w0 + piece : words;
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

cudaError_t launch_fetch(const FetchArgs& a, int blocks, cudaStream_t s) {
  prof_begin(kProfFetch, s);
  fetch_kernel<<<blocks, 256, 0, s>>>(a);
  prof_end(kProfFetch, s);
  return cudaGetLastError();
}

cudaError_t launch_cache_step(const CacheStepArgs& a, cudaStream_t s) {
  prof_begin(kProfCache, s);
  cache_step_kernel<<<1, 32, 0, s>>>(a);
  prof_end(kProfCache, s);
  return cudaGetLastError();
}

}  // namespace mcft
