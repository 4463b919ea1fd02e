// LoRA down-projections for the Stage-2 expert forward (Section 3.2: the experts are fine-tuned
// with LoRA adapters; rank 8 and alpha 16 in Appendix B).
//
// Each adapted projection is W v + s B (A v) with A [r, in], B [out, r], s = alpha / r. The large
// term W v runs in the expert GEMM / GEMV kernels, which also add s B u in their epilogues (r
// multiply-adds per output). On the decode and fp32 paths this kernel computes the small middle
// vectors u = A v for every permuted row whose segment has an adapter (the tcgen05 path projects
// its gathered rows on the tensor cores and takes A2 h from GEMM13's epilogue instead):
//   stage 13: u[q] = [A1 x ; A3 x]     (2r values; x = the row's token, or the gathered row)
//   stage 2:  u[q] = A2 h_q            (r values; h = the SwiGLU activation of the row)
// One warp per row: lanes walk the input in 16-byte chunks, each chunk is dotted with the R rows
// of A (small, L1/L2-resident), and R warp reductions finish the row. Rows of segments without an
// adapter, and padding rows, get zeros.
#include "common.cuh"
#include "internal.h"

namespace mcft {
namespace {

constexpr int kWarps = 8;

template <typename T>
struct In16;  // 16 bytes of an input or adapter row as fp32
template <>
struct In16<__nv_bfloat16> {
  static constexpr int n = 8;
  __device__ static void load(const void* p, float* f) { unpack8(ldg16(p), f); }
};
template <>
struct In16<float> {
  static constexpr int n = 4;
  __device__ static void load(const void* p, float* f) {
    const uint4 v = ldg16(p);
    f[0] = __uint_as_float(v.x); f[1] = __uint_as_float(v.y);
    f[2] = __uint_as_float(v.z); f[3] = __uint_as_float(v.w);
  }
};

// T: dtype of the input rows and of the adapter (the layer dtype); R: outputs per row (2r or r).
template <typename T, int R>
__global__ void __launch_bounds__(kWarps * 32) lora_down_kernel(const __grid_constant__ LoraDownArgs a) {
  pdl_wait();
  __shared__ int s_off[kMaxSeg + 1];
  __shared__ int s_nseg;
  if (threadIdx.x == 0) s_nseg = a.hdr->abort == 0 ? a.nseg : 0;
  __syncthreads();
  const int nseg = s_nseg;
  for (int s = threadIdx.x; s <= nseg; s += blockDim.x) s_off[s] = a.off[s];
  __syncthreads();
  if (nseg == 0) return;
  const int mrows = s_off[nseg];
  const int lane = threadIdx.x & 31;
  using C = In16<T>;
  for (int q = blockIdx.x * kWarps + (threadIdx.x >> 5); q < mrows; q += gridDim.x * kWarps) {
    int s = 0;
    while (s + 1 < nseg && s_off[s + 1] <= q) ++s;
    const char* blk = reinterpret_cast<const char*>(a.lblk[s]);
    const int tok = a.row_tok[q];  // -1 for a padding row
    float* out = a.u + size_t(q) * a.ustride;
    if (blk == nullptr || tok < 0) {
      for (int j = lane; j < R; j += 32) out[j] = 0.f;
      continue;
    }
    const int src = a.by_token ? tok : q;  // x is indexed by token, h by permuted row
    const char* in = reinterpret_cast<const char*>(a.in) + size_t(src) * a.in_stride * sizeof(T);
    float acc[R];
#pragma unroll
    for (int j = 0; j < R; ++j) acc[j] = 0.f;
    for (int k = lane * C::n; k < a.K; k += 32 * C::n) {
      float xv[C::n];
      C::load(in + size_t(k) * sizeof(T), xv);
#pragma unroll
      for (int j = 0; j < R; ++j) {
        // adapter row j: rows of the first A (A1 or A2), then of the second (A3) at stage 13
        const size_t aoff = j < a.r ? a.a_off0 + size_t(j) * a.K : a.a_off1 + size_t(j - a.r) * a.K;
        float wv[C::n];
        C::load(blk + (aoff + k) * sizeof(T), wv);
#pragma unroll
        for (int i = 0; i < C::n; ++i) acc[j] = fmaf(wv[i], xv[i], acc[j]);
      }
    }
#pragma unroll
    for (int j = 0; j < R; ++j) {
      const float v = warp_sum(acc[j]);
      if (lane == 0) out[j] = v;
    }
  }
}

template <typename T>
cudaError_t launch_typed(const LoraDownArgs& a, int outs, int blocks, cudaStream_t s) {
  switch (outs) {
    case 8: lora_down_kernel<T, 8><<<blocks, kWarps * 32, 0, s>>>(a); break;
    case 16: lora_down_kernel<T, 16><<<blocks, kWarps * 32, 0, s>>>(a); break;
    case 32: lora_down_kernel<T, 32><<<blocks, kWarps * 32, 0, s>>>(a); break;
    default: return cudaErrorInvalidValue;
  }
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_lora_down(const LoraDownArgs& a, int dtype, int outs, int mcap, cudaStream_t s) {
  int blocks = (mcap + kWarps - 1) / kWarps;
  if (blocks > 4096) blocks = 4096;
  if (blocks < 1) blocks = 1;
  prof_begin(kProfLora, s);
  const cudaError_t e = dtype == MCFT_BF16 ? launch_typed<__nv_bfloat16>(a, outs, blocks, s)
                                           : launch_typed<float>(a, outs, blocks, s);
  prof_end(kProfLora, s);
  return e;
}

}  // namespace mcft
