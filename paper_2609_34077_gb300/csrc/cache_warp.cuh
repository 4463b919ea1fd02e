// Per-layer expert cache decisions as warp-level device functions (Section 4.1 "Simulation",
// Eq. metrics): the cache step and the prefetch event. Each runs on one warp of a CTA; the standalone
// kernels of cache.cu and the fused decode prologue of prologue.cu call the same code, so both
// paths make identical decisions. The rules are stated in cache.cu.
#pragma once

#include "common.cuh"
#include "internal.h"

namespace mcft {

// Slot for an expert that enters at time stamp t, chosen by the whole warp (every lane returns the
// same slot): the lowest free slot, else the victim among the slots not used at t, else -1. The
// victim has the smallest key of the policy: (access count of its expert, last use, expert id) for
// LFU, (last use, expert id) for LRU, (insertion, expert id) for FIFO, found by a warp arg-min over
// one key per slot. Stamps of occupied slots are >= 0 and ids < 64, so a stamp and an id pack into
// one 64-bit word; ids are distinct, so the minimum is unique.
__device__ __forceinline__ int warp_pick_slot(int policy, int B, int64_t t, const int32_t* tag,
                                              const int64_t* last, const int64_t* ins,
                                              const int64_t* freq) {
  const unsigned full = 0xffffffffu;
  const int lane = threadIdx.x & 31;
  const unsigned f0 = __ballot_sync(full, lane < B && tag[lane] < 0);
  const unsigned f1 = __ballot_sync(full, lane + 32 < B && tag[lane + 32] < 0);
  if (f0) return __ffs(f0) - 1;
  if (f1) return 32 + __ffs(f1) - 1;
  unsigned long long hi = ~0ull, lo = ~0ull;
  int slot = -1;
  for (int j = 0; j < 2; ++j) {
    const int sl = lane + 32 * j;
    if (sl < B && last[sl] < t) {  // no free slot: tag[sl] >= 0
      const unsigned long long e = static_cast<unsigned long long>(tag[sl]);
      const unsigned long long h =
          policy == MCFT_CACHE_LFU ? static_cast<unsigned long long>(freq[e]) : 0ull;
      const unsigned long long l =
          (static_cast<unsigned long long>(policy == MCFT_CACHE_FIFO ? ins[sl] : last[sl]) << 8) | e;
      if (h < hi || (h == hi && l < lo)) {
        hi = h;
        lo = l;
        slot = sl;
      }
    }
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const unsigned long long h2 = __shfl_xor_sync(full, hi, o), l2 = __shfl_xor_sync(full, lo, o);
    const int s2 = __shfl_xor_sync(full, slot, o);
    if (h2 < hi || (h2 == hi && l2 < lo)) {
      hi = h2;
      lo = l2;
      slot = s2;
    }
  }
  return slot;
}

__device__ inline void cache_step_warp(const CacheStepArgs& a) {
  __shared__ int32_t s_tag[kMaxE];
  __shared__ int64_t s_last[kMaxE], s_ins[kMaxE], s_freq[kMaxE];
  __shared__ int32_t s_out[1 + 3 * kMaxE];  // n_miss, miss experts, miss locations, loc_of
  const int lane = threadIdx.x & 31;
  const int B = a.B, E = a.E;
  // every global load of the step is issued up front (the layer's step and prefetch mask, then
  // its slot state below), so the warp pays about one round trip for them, not one each
  const int64_t t = a.step[a.layer];
  const unsigned long long pf_in = a.pfmask[a.layer];
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
      if (a.stream) *a.stream = 0;
      if (a.fctr) a.fctr[0] = a.fctr[1] = 0u;
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
  // the replacement rule, warp-parallel over slots; misses one at a time in ascending id
  int32_t* m_exp = s_out + 1;
  int32_t* m_loc = s_out + 1 + E;
  int32_t* loc_of = s_out + 1 + 2 * E;
  const unsigned long long pf = pf_in;
  const unsigned long long drop = pf & ~mine;  // prefetched experts this step does not use
  for (int e = lane; e < E; e += 32) loc_of[e] = -1;
  for (int sl = lane; sl < B; sl += 32) {
    const int e = s_tag[sl];
    if (e >= 0 && ((drop >> e) & 1ull)) {
      s_tag[sl] = -1;
      s_last[sl] = -1;
      s_ins[sl] = -1;
    }
  }
  if (lane == 0) a.cancel[a.layer] = drop;
  __syncwarp();
  unsigned long long cached = 0;
  int hits = 0;
  for (int sl = lane; sl < B; sl += 32) {
    const int e = s_tag[sl];
    if (e < 0) continue;
    cached |= 1ull << e;
    if ((mine >> e) & 1ull) {
      s_last[sl] = t;
      loc_of[e] = sl;
      ++hits;
    }
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    cached |= __shfl_xor_sync(0xffffffffu, cached, o);
    hits += __shfl_xor_sync(0xffffffffu, hits, o);
  }
  __syncwarp();
  const int useful = __popcll(pf & mine & cached);
  unsigned long long miss = mine & ~cached;
  int nm = 0, nbyp = 0;
  while (miss) {
    const int e = __ffsll(static_cast<long long>(miss)) - 1;  // ascending expert id
    miss &= miss - 1;
    const int slot = warp_pick_slot(a.policy, B, t, s_tag, s_last, s_ins, s_freq);
    __syncwarp();
    if (lane == 0) {
      m_exp[nm] = e;
      if (slot < 0) {
        m_loc[nm] = -1;
        loc_of[e] = B + nbyp;
      } else {
        s_tag[slot] = e;
        s_last[slot] = t;
        s_ins[slot] = t;
        m_loc[nm] = slot;
        loc_of[e] = slot;
      }
    }
    if (slot < 0) ++nbyp;
    ++nm;
    __syncwarp();  // the next pick sees this slot taken
  }
  if (lane == 0) {
    s_out[0] = nm;
    a.step[a.layer] = t + 1;
    unsigned long long* c = a.counters + size_t(a.layer) * kCacheCounters;
    atomicAdd(c + 0, static_cast<unsigned long long>(hits));  // no value returned: no round trip
    atomicAdd(c + 1, static_cast<unsigned long long>(nm));
    atomicAdd(c + 2, static_cast<unsigned long long>(nbyp));
    atomicAdd(c + 4, static_cast<unsigned long long>(useful));
    a.pfmask[a.layer] = 0;
  }
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
  if (lane == 0) {
    *a.ready = hitbits;
    // the misses, which this step's demand fetch copies (none without slots)
    if (a.stream) *a.stream = a.slots ? (mine & ~cached) : 0ull;
    if (a.fctr) a.fctr[0] = a.fctr[1] = 0u;  // for the FFN launch that fetches these misses
  }
  // No fence: the FFN and fetch kernels read these after a kernel boundary (or an event), the host
  // after synchronising on one; the running fetch kernel that polls the cancel mask only needs the
  // write to arrive, in any order.
}

// Prefetch decision (one warp). The lanes count how many predicted (token, k) entries name each
// expert, touch the cached candidates and rank the uncached ones (warp max over packed keys); the
// loads then claim slots in ascending id (each slot a warp-wide choice) and the lanes write the
// fetch list.
__device__ inline void prefetch_warp(const PrefetchArgs& a) {
  __shared__ int cnt[kMaxE], rank[kMaxE];
  __shared__ int32_t s_tag[kMaxE];
  __shared__ int64_t s_last[kMaxE], s_ins[kMaxE], s_freq[kMaxE];
  __shared__ int32_t s_list[1 + kMaxE];
  const int lane = threadIdx.x & 31, B = a.B, E = a.E;
  // the layer's step and prefetch mask are loaded up front, beside the slot state below
  const int64_t t = a.step[a.layer];
  const unsigned long long pf_in = a.pfmask[a.layer];
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
  // every cached candidate is touched; the loads are the n_max best-ranked uncached candidates by
  // (count descending, best rank ascending, id ascending): warp-parallel sets and a warp max over
  // one packed key per expert
  unsigned long long cand = 0, cached = 0, load = 0;
  for (int e = lane; e < E; e += 32)
    if (cnt[e] > 0) cand |= 1ull << e;
  for (int sl = lane; sl < B; sl += 32)
    if (s_tag[sl] >= 0) cached |= 1ull << s_tag[sl];
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    cand |= __shfl_xor_sync(0xffffffffu, cand, o);
    cached |= __shfl_xor_sync(0xffffffffu, cached, o);
  }
  for (int sl = lane; sl < B; sl += 32)
    if (s_tag[sl] >= 0 && ((cand >> s_tag[sl]) & 1ull)) s_last[sl] = t;
  for (int j = 0; j < a.n_max; ++j) {
    unsigned key = 0;  // 0 = nothing left
    for (int e = lane; e < E; e += 32)
      if (((cand & ~cached & ~load) >> e) & 1ull) {
        const unsigned c = cnt[e] < 32767 ? unsigned(cnt[e]) : 32767u;
        const unsigned k = (c << 16) | ((255u - unsigned(rank[e])) << 8) | (255u - unsigned(e));
        key = key > k ? key : k;
      }
    key = __reduce_max_sync(0xffffffffu, key);
    if (key == 0) break;
    load |= 1ull << (255u - (key & 255u));
  }
  __syncwarp();
  // slots for the loads, one at a time in ascending id (warp-parallel choice of each slot)
  unsigned long long pf = pf_in;
  int nl = 0;
  while (load) {
    const int e = __ffsll(static_cast<long long>(load)) - 1;
    load &= load - 1;
    const int slot = warp_pick_slot(a.policy, B, t, s_tag, s_last, s_ins, s_freq);
    if (slot < 0) continue;  // unreachable with n_max <= B; kept for safety
    const int old = s_tag[slot];
    if (old >= 0) pf &= ~(1ull << old);
    pf |= 1ull << e;
    __syncwarp();  // every lane has read the slot before lane 0 rewrites it
    if (lane == 0) {
      s_tag[slot] = e;
      s_last[slot] = t;
      s_ins[slot] = t;
      s_list[1 + nl] = e;
    }
    ++nl;
    __syncwarp();
  }
  if (lane == 0) {
    s_list[0] = nl;
    a.pfmask[a.layer] = pf;
    a.cancel[a.layer] = 0;
    a.step[a.layer] = t + 1;
    atomicAdd(a.counters + size_t(a.layer) * kCacheCounters + 3, static_cast<unsigned long long>(nl));
  }
  __syncwarp();
  for (int i = lane; i < B; i += 32) {
    tag[i] = s_tag[i];
    last[i] = s_last[i];
    ins[i] = s_ins[i];
  }
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

}  // namespace mcft
