// Router GEMV + mask / prior + Top-K + gate softmax, one CTA per token.
//
// z = W x (Section 3.1); the score is z (plain Top-K, Eq. topk), z restricted to m_e = 1 (hard
// mask, Eq. stage1) or z_e + log pi_e (soft prior, Eq. inference: log(p_e pi_e) = z_e + log pi_e
// - logsumexp(z), the same order as p_e pi_e). The K best scores are taken largest first, equal
// scores to the lower expert index. Gates come from p = softmax(z): renormalised over the active
// set (Mixtral) or p_i itself (DeepSeek).
//
// Layout: 8 warps split d; each lane keeps one fp32 partial sum per expert; warps combine through
// shared memory; warp 0 ranks (two experts per lane, shuffle arg-max) and writes idx / gate.
#include "common.cuh"
#include "internal.h"

namespace mcft {
namespace {

constexpr int kWarps = 8;

template <typename TX>
struct Chunk;  // 16 bytes of a row: 8 bf16 or 4 fp32
template <>
struct Chunk<__nv_bfloat16> {
  static constexpr int n = 8;
  __device__ static void load(const void* p, float* f) { unpack8(ldg16(p), f); }
};
template <>
struct Chunk<float> {
  static constexpr int n = 4;
  __device__ static void load(const void* p, float* f) {
    uint4 v = ldg16(p);
    f[0] = __uint_as_float(v.x); f[1] = __uint_as_float(v.y);
    f[2] = __uint_as_float(v.z); f[3] = __uint_as_float(v.w);
  }
};

// Warp arg-max over (value, index) with ties to the lower index; ineligible = -inf and index E.
__device__ __forceinline__ void warp_argmax(float& v, int& i) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    float v2 = __shfl_xor_sync(0xffffffffu, v, o);
    int i2 = __shfl_xor_sync(0xffffffffu, i, o);
    if (v2 > v || (v2 == v && i2 < i)) { v = v2; i = i2; }
  }
}

template <typename TX, int MAXE>
__global__ void __launch_bounds__(kWarps * 32) route_kernel(const __grid_constant__ RouteArgs a) {
  __shared__ float part[kWarps][MAXE];
  __shared__ float zs[MAXE];
  const int t = blockIdx.x;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int E = a.E, d = a.d;
  using C = Chunk<TX>;
  const int nchunk = d / C::n;

  float acc[MAXE];
#pragma unroll
  for (int e = 0; e < MAXE; ++e) acc[e] = 0.f;

  const char* xrow = reinterpret_cast<const char*>(a.x) + size_t(t) * d * sizeof(TX);
  const char* wr = reinterpret_cast<const char*>(a.w_router);
  const size_t wrow = size_t(d) * sizeof(TX);
  for (int c = warp * 32 + lane; c < nchunk; c += kWarps * 32) {
    float xv[C::n];
    C::load(xrow + size_t(c) * 16, xv);
#pragma unroll
    for (int e = 0; e < MAXE; ++e) {
      if (e < E) {
        float wv[C::n];
        C::load(wr + e * wrow + size_t(c) * 16, wv);
#pragma unroll
        for (int j = 0; j < C::n; ++j) acc[e] = fmaf(xv[j], wv[j], acc[e]);
      }
    }
  }
#pragma unroll
  for (int e = 0; e < MAXE; ++e) {
    if (e < E) {
      float v = warp_sum(acc[e]);
      if (lane == 0) part[warp][e] = v;
    }
  }
  __syncthreads();
  if (warp != 0) return;
  for (int e = lane; e < E; e += 32) {
    float v = 0.f;
#pragma unroll
    for (int w = 0; w < kWarps; ++w) v += part[w][e];
    zs[e] = v;
  }
  __syncwarp();

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

template <typename TX>
cudaError_t launch_typed(const RouteArgs& a, cudaStream_t s) {
  dim3 grid(a.T), block(kWarps * 32);
  prof_begin(kProfRoute, s);
  if (a.E <= 8) route_kernel<TX, 8><<<grid, block, 0, s>>>(a);
  else if (a.E <= 16) route_kernel<TX, 16><<<grid, block, 0, s>>>(a);
  else if (a.E <= 32) route_kernel<TX, 32><<<grid, block, 0, s>>>(a);
  else route_kernel<TX, 64><<<grid, block, 0, s>>>(a);
  prof_end(kProfRoute, s);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_route(const RouteArgs& a, int dtype, cudaStream_t s) {
  if (a.T == 0) return cudaSuccess;
  return dtype == MCFT_BF16 ? launch_typed<__nv_bfloat16>(a, s) : launch_typed<float>(a, s);
}

}  // namespace mcft
