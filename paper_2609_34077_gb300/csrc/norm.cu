// Residual stream of the chained decode stack: x_{l+1} = x_l + y_l, and the RMS-normalised input of
// the next MoE block, u = gamma * x / sqrt(mean_j x[j]^2 + eps) (the block-input norm of Mixtral and
// DeepSeek-V2; the paper's models, Section 4 and Table 4).
//
// One CTA of 256 threads per token row. Each thread owns the same 4-element groups in both passes
// (so it reads back what it wrote itself); the sum of squares is reduced in a fixed order (warp
// shuffle tree, then the 8 warp sums in order), so the result does not depend on scheduling. The
// stream stays fp32; u is stored in the layer dtype (bf16 rounding to nearest even).
#include "common.cuh"
#include "internal.h"

namespace mcft {
namespace {

template <typename T>
__device__ __forceinline__ float4 load4(const void* p, size_t i) {
  if constexpr (sizeof(T) == 2) {
    const uint2 v = *reinterpret_cast<const uint2*>(reinterpret_cast<const uint16_t*>(p) + i);
    return make_float4(bf16lo(v.x), bf16hi(v.x), bf16lo(v.y), bf16hi(v.y));
  } else {
    return *reinterpret_cast<const float4*>(reinterpret_cast<const float*>(p) + i);
  }
}

template <typename T>
__device__ __forceinline__ void store4(void* p, size_t i, float4 v) {
  if constexpr (sizeof(T) == 2) {
    *reinterpret_cast<uint2*>(reinterpret_cast<uint16_t*>(p) + i) =
        make_uint2(pack2bf(v.x, v.y), pack2bf(v.z, v.w));
  } else {
    *reinterpret_cast<float4*>(reinterpret_cast<float*>(p) + i) = v;
  }
}

template <typename T>
__global__ void __launch_bounds__(256) resid_norm_kernel(const __grid_constant__ NormArgs a) {
  pdl_wait();
  __shared__ float part[8];
  const size_t row = size_t(blockIdx.x) * a.d;
  float* x = a.x + row;
  float ss = 0.f;
  for (int c = threadIdx.x * 4; c < a.d; c += 1024) {
    float4 v = *reinterpret_cast<const float4*>(x + c);
    if (a.y) {
      const float4 y = load4<T>(a.y, row + c);
      v.x += y.x; v.y += y.y; v.z += y.z; v.w += y.w;
      *reinterpret_cast<float4*>(x + c) = v;
    }
    ss = fmaf(v.x, v.x, ss);
    ss = fmaf(v.y, v.y, ss);
    ss = fmaf(v.z, v.z, ss);
    ss = fmaf(v.w, v.w, ss);
  }
  if (!a.gamma) return;
  ss = warp_sum(ss);
  if ((threadIdx.x & 31) == 0) part[threadIdx.x >> 5] = ss;
  __syncthreads();
  float tot = 0.f;
#pragma unroll
  for (int w = 0; w < 8; ++w) tot += part[w];
  const float r = 1.0f / sqrtf(tot / float(a.d) + a.eps);
  for (int c = threadIdx.x * 4; c < a.d; c += 1024) {
    const float4 v = *reinterpret_cast<const float4*>(x + c);
    const float4 g = load4<T>(a.gamma, c);
    store4<T>(a.u, row + c, make_float4(v.x * r * g.x, v.y * r * g.y, v.z * r * g.z, v.w * r * g.w));
  }
}

}  // namespace

cudaError_t launch_resid_norm(const NormArgs& a, int dtype, cudaStream_t s) {
  prof_begin(kProfNorm, s);
  const cudaError_t e = dtype == MCFT_BF16
      ? launch_pdl(resid_norm_kernel<uint16_t>, dim3(a.T), dim3(256), 0, s, a)
      : launch_pdl(resid_norm_kernel<float>, dim3(a.T), dim3(256), 0, s, a);
  prof_end(kProfNorm, s);
  return e != cudaSuccess ? e : cudaGetLastError();
}

}  // namespace mcft
