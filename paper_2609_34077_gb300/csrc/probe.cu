// HBM read probe (mcft_read_probe): how long one launch of the decode FFN's grid takes to read a
// buffer, with no computation on the data. Measurement infrastructure with no counterpart in the
// paper: the decode FFN's rooflines are taken against the measured copy peak, and this shows what
// a launch of the same shape can read at all, as a contiguous stream or with exactly the FFN's
// weight-load pattern. Every 32-bit word is read once and folded into one XOR per thread, and the
// threads' XORs are combined in *sink, so a caller can check that every byte was read.
#include "common.cuh"
#include "internal.h"

namespace mcft {
namespace {

__device__ __forceinline__ unsigned fold(const uint4& v) { return v.x ^ v.y ^ v.z ^ v.w; }

// One contiguous stream: grid-strided 16-byte loads, eight in flight per thread.
__global__ void __launch_bounds__(256, 2) read_contiguous_kernel(const uint4* __restrict__ p,
                                                                 size_t n16, unsigned* sink) {
  pdl_wait();
  const size_t nth = size_t(gridDim.x) * blockDim.x;
  size_t i = size_t(blockIdx.x) * blockDim.x + threadIdx.x;
  unsigned acc = 0;
  for (; i + 7 * nth < n16; i += 8 * nth) {
    uint4 v[8];
#pragma unroll
    for (int j = 0; j < 8; ++j) v[j] = ld_stream16(p + i + j * nth);
#pragma unroll
    for (int j = 0; j < 8; ++j) acc ^= fold(v[j]);
  }
  for (; i < n16; i += nth) acc ^= fold(ld_stream16(p + i));
  if (acc != 0u) atomicXor(sink, acc);
}

// The decode FFN's GEMM13 load pattern: items of 32 rows (16 W1 rows, then 16 W3 rows of a row
// block), items strided over the grid; warp w reads the 128-byte chunks w, w + 8, ... of every row
// of the item, a lane of quad position c the bytes 16c .. 16c + 15 and 64 + 16c .. 64 + 16c + 15
// of rows g, g + 8, g + 16, g + 24 (g = lane / 4): eight 16-byte loads per lane per step.
__global__ void __launch_bounds__(256, 2) read_rows_kernel(const char* __restrict__ p,
                                                           size_t nitems, int rowb, unsigned* sink) {
  pdl_wait();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int g = lane >> 2, c = lane & 3;
  const size_t item_bytes = size_t(32) * rowb;
  const int nch = rowb / 128;
  unsigned acc = 0;
  for (size_t it = blockIdx.x; it < nitems; it += gridDim.x) {
    const char* b = p + it * item_bytes + c * 16;
    for (int ch = warp; ch < nch; ch += 8) {
      const char* r = b + size_t(g) * rowb + size_t(ch) * 128;
      uint4 v[8];
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        v[2 * q] = ld_stream16(r + size_t(8 * q) * rowb);
        v[2 * q + 1] = ld_stream16(r + size_t(8 * q) * rowb + 64);
      }
#pragma unroll
      for (int j = 0; j < 8; ++j) acc ^= fold(v[j]);
    }
  }
  if (acc != 0u) atomicXor(sink, acc);
}

}  // namespace

cudaError_t launch_read_probe(const void* buf, size_t bytes, int pattern, int row_bytes,
                              int blocks, unsigned* sink, cudaStream_t s) {
  if (pattern == 0)
    return launch_pdl(read_contiguous_kernel, dim3(blocks), dim3(256), 0, s,
                      static_cast<const uint4*>(buf), bytes / 16, sink);
  return launch_pdl(read_rows_kernel, dim3(blocks), dim3(256), 0, s, static_cast<const char*>(buf),
                    bytes / (size_t(32) * row_bytes), row_bytes, sink);
}

}  // namespace mcft
