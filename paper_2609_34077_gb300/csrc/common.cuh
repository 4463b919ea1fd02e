// Shared device helpers for libmcft (sm_103a). Not part of the C ABI.
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

namespace mcft {

constexpr int kMaxE = 64;        // routed experts per layer
constexpr int kMaxK = 8;         // active experts per token
constexpr int kMaxShared = 8;    // shared experts per layer
constexpr int kMaxSeg = kMaxE + kMaxShared;

// Device error codes (same values as mcft_status).
constexpr unsigned kErrInvalid = 1u;
constexpr unsigned kErrTimeout = 4u;

// Record the first device-side error; later ones keep the first code.
__device__ __forceinline__ void set_error(unsigned* err, unsigned code) {
  if (err) atomicCAS(err, 0u, code);
}

// 16-byte vector of weights or activations.
struct alignas(16) V16 {
  uint4 u;
};

// Programmatic dependent launch: a kernel launched with programmatic stream serialization may
// start while the previous kernel of its stream is still finishing; this wait returns once that
// kernel has completed and its memory operations are visible. Every kernel of the library calls
// it before its first global memory access (a no-op for kernels launched without the attribute).
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }

__device__ __forceinline__ uint4 ldg16(const void* p) {
  return __ldg(reinterpret_cast<const uint4*>(p));
}

// 16-byte load through L2 only (coherent with stores of other CTAs of the same kernel that were
// published with a fence: no stale L1 line can be returned).
__device__ __forceinline__ uint4 ldcg16(const void* p) {
  uint4 r;
  asm volatile("ld.global.cg.v4.u32 {%0,%1,%2,%3}, [%4];"
               : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w)
               : "l"(p));
  return r;
}

// Streaming (read-once) 16-byte load: do not keep in L1.
__device__ __forceinline__ uint4 ld_stream16(const void* p) {
  uint4 r;
  asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
               : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w)
               : "l"(p));
  return r;
}

__device__ __forceinline__ float bf16lo(uint32_t v) { return __uint_as_float(v << 16); }
__device__ __forceinline__ float bf16hi(uint32_t v) { return __uint_as_float(v & 0xffff0000u); }

// Unpack 8 bf16 held in a uint4 into fp32.
__device__ __forceinline__ void unpack8(const uint4& v, float* f) {
  f[0] = bf16lo(v.x); f[1] = bf16hi(v.x);
  f[2] = bf16lo(v.y); f[3] = bf16hi(v.y);
  f[4] = bf16lo(v.z); f[5] = bf16hi(v.z);
  f[6] = bf16lo(v.w); f[7] = bf16hi(v.w);
}

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

// Round fp32 to bf16 (round to nearest even) and back to its bit pattern.
__device__ __forceinline__ uint16_t f2bf(float f) {
  __nv_bfloat16 b = __float2bfloat16_rn(f);
  return *reinterpret_cast<uint16_t*>(&b);
}

__device__ __forceinline__ uint32_t pack2bf(float a, float b) {
  return uint32_t(f2bf(a)) | (uint32_t(f2bf(b)) << 16);
}

// One piece [w0, w1) of a host-to-device copy, in 16-byte words, by the whole CTA: each thread
// keeps four loads in flight before it stores them (64 KB outstanding per 256-thread CTA).
__device__ __forceinline__ void copy_piece(const uint4* src, uint4* dst, size_t w0, size_t w1) {
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

// D += A B on the tensor cores, one warp: A 16 x 16 bf16 (row), B 16 x 8 bf16 (col), D fp32.
__device__ __forceinline__ void mma16816(float* d, uint32_t a0, uint32_t a1, uint32_t a2,
                                         uint32_t a3, uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, "
      "{%8,%9}, {%0,%1,%2,%3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

__device__ __forceinline__ float silu(float u) { return u / (1.0f + expf(-u)); }

__device__ __forceinline__ uint64_t globaltimer_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %globaltimer;" : "=l"(t));
  return t;
}

}  // namespace mcft
