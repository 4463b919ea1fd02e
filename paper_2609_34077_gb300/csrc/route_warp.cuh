// Top-K under a mask or a soft prior and the gate weights of one token, from its router logits
// (Section 3.1 Eq. topk; Section 3.2 Eq. stage1 and Eq. inference), as a warp-level device function.
// The router kernel (route.cu) and the fused decode prologue (prologue.cu) both call it, so both
// rank identically: the K best scores largest first, equal scores to the lower expert index
// (z_e under a hard mask, z_e + log pi_e under a soft prior); gates from p = softmax(z),
// renormalised over the active set (Mixtral) or p_i itself (DeepSeek).
#pragma once

#include "common.cuh"
#include "internal.h"

namespace mcft {

// Warp arg-max over (value, index) with ties to the lower index; ineligible = -inf and index E.
__device__ __forceinline__ void warp_argmax(float& v, int& i) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    float v2 = __shfl_xor_sync(0xffffffffu, v, o);
    int i2 = __shfl_xor_sync(0xffffffffu, i, o);
    if (v2 > v || (v2 == v && i2 < i)) { v = v2; i = i2; }
  }
}

// Called by one whole warp: zs = the token's E router logits (shared memory), t = its row in
// a.idx / a.gate.
__device__ inline void rank_and_gate_warp(const RouteArgs& a, const float* zs, int t) {
  const int lane = threadIdx.x & 31, E = a.E;
  // Each lane owns experts lane and lane + 32.
  float z[2], s[2];
  bool elig[2];
#pragma unroll
  for (int j = 0; j < 2; ++j) {
    const int e = lane + 32 * j;
    elig[j] = e < E;
    z[j] = elig[j] ? zs[e] : -INFINITY;
    s[j] = z[j];
    if (elig[j]) {
      if (a.mode == MCFT_ROUTE_HARD_MASK) {
        elig[j] = a.mask[e] != 0;
      } else if (a.mode == MCFT_ROUTE_SOFT_PRIOR) {
        s[j] = z[j] + logf(a.prior[e]);
      }
      if (s[j] != s[j]) {  // NaN input
        set_error(a.err, kErrInvalid);
        elig[j] = false;
      }
    }
  }
  int sel_k[2] = {-1, -1};  // rank at which this lane's expert was selected
  float zsel = 0.f;
  int isel = 0;
  for (int k = 0; k < a.K; ++k) {
    float v = -INFINITY;
    int i = 1 << 30;
#pragma unroll
    for (int j = 0; j < 2; ++j) {
      const int e = lane + 32 * j;
      if (elig[j] && sel_k[j] < 0 && (s[j] > v || (s[j] == v && e < i) || i == (1 << 30))) {
        v = s[j];
        i = e;
      }
    }
    warp_argmax(v, i);
#pragma unroll
    for (int j = 0; j < 2; ++j)
      if (lane + 32 * j == i) sel_k[j] = k;
    if (i >= E) {  // fewer eligible experts than K: only reachable through NaN inputs
      set_error(a.err, kErrInvalid);
      i = 0;
    }
    if (lane == k) isel = i;
  }
  if (lane < a.K) zsel = zs[isel];
  // gate softmax from z (p = softmax(z) over all E; renormalised over A or not)
  float m, den;
  if (a.gate_mode == MCFT_GATE_RENORM) {
    m = lane < a.K ? zsel : -INFINITY;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, o));
    den = warp_sum(lane < a.K ? expf(zsel - m) : 0.f);
  } else {
    m = fmaxf(z[0], z[1]);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, o));
    float ex = 0.f;
#pragma unroll
    for (int j = 0; j < 2; ++j)
      if (lane + 32 * j < E) ex += expf(z[j] - m);
    den = warp_sum(ex);
  }
  if (lane < a.K) {
    a.idx[size_t(t) * a.K + lane] = isel;
    a.gate[size_t(t) * a.K + lane] = expf(zsel - m) / den;
  }
}

}  // namespace mcft
