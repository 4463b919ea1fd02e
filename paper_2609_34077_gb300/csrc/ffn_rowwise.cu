// Row-streaming expert FFN for fp32 layers (CUDA-core fp32 arithmetic), plus the combine.
//
// F(x) = W2 (silu(W1 x) * (W3 x)) per expert segment (Section 3.1; SwiGLU experts). Each weight
// row is read once per call from HBM with 16-byte loads and dotted with every token of its segment
// (up to 8 at a time from L1), so the kernel streams the selected experts' weights at the rate of
// the memory system when segments hold few tokens. Work items are (segment, 16-row block), spread
// over a persistent grid sized to the SMs.
//
// combine: y[t] = sum_k gate[t,k] o[pos(t,k)] + sum_s o[shared row of t in segment E+s], summed in
// k order then shared-expert order (deterministic).
#include <type_traits>

#include "common.cuh"
#include "internal.h"

namespace mcft {
namespace {

constexpr int kWarps = 8;
constexpr int kRowsPerWarp = 2;
constexpr int kRowsPerItem = kWarps * kRowsPerWarp;
constexpr int kTokGroup = 8;

template <typename TW>
struct W16;  // one 16-byte chunk of a row
template <>
struct W16<__nv_bfloat16> {
  static constexpr int n = 8;
  __device__ static void cvt(const uint4& v, float* f) { unpack8(v, f); }
};
template <>
struct W16<float> {
  static constexpr int n = 4;
  __device__ static void cvt(const uint4& v, float* f) {
    f[0] = __uint_as_float(v.x); f[1] = __uint_as_float(v.y);
    f[2] = __uint_as_float(v.z); f[3] = __uint_as_float(v.w);
  }
};

struct Items {
  int nseg, total;
  int off[kMaxSeg + 1];
  int first[kMaxSeg + 1];  // first item of each segment
  const char* blk[kMaxSeg];
};

// Prefix of work items over non-empty segments (rows_per_seg / kRowsPerItem items each).
__device__ void build_items(Items& it, const FfnArgs& a, int rows_per_seg) {
  if (threadIdx.x == 0) {
    const int nseg = a.hdr->abort == 0 ? a.nseg : 0;
    it.nseg = nseg;
    int acc = 0;
    const unsigned long long hits = a.ready ? *a.ready : 0ull;
    for (int s = 0; s <= nseg; ++s) it.off[s] = a.off[s];
    for (int s = 0; s < nseg; ++s) {
      it.first[s] = acc;
      it.blk[s] = reinterpret_cast<const char*>(seg_block(a, s));
      const int n = it.off[s + 1] - it.off[s];
      if (n > 0 && seg_in_phase(a, s, hits)) {
        if (it.blk[s] == nullptr) {  // a selected expert without weights
          set_error(a.err, kErrInvalid);
          const_cast<WsHeader*>(a.hdr)->abort = 1;
          continue;
        }
        acc += rows_per_seg / kRowsPerItem;
      }
    }
    it.first[nseg] = acc;
    it.total = acc;
  }
  __syncthreads();
}

__device__ __forceinline__ int find_seg(const Items& it, int item) {
  int s = 0;
  // the last segment whose first item is <= item; it is never empty (its end lies past item)
  while (s + 1 < it.nseg && it.first[s + 1] <= item) ++s;
  return s;
}

// h[q, r] = silu(W1[r] . x_t) * (W3[r] . x_t) for rows r = r0, r0 + 1 and NT tokens of a segment.
template <typename TW, int NT>
__device__ __forceinline__ void ffn13_tile(const FfnArgs& a, const char* blk, const void* lblk,
                                           int r0, int q0, int nt, const int* tok, int lane) {
  using C = W16<TW>;
  const size_t rowb = size_t(a.d) * sizeof(TW);
  const char* w1a = blk + size_t(r0) * rowb;
  const char* w1b = w1a + rowb;
  const char* w3a = blk + size_t(a.w + r0) * rowb;
  const char* w3b = w3a + rowb;
  const char* xb = reinterpret_cast<const char*>(a.x);
  const char* xr[NT];
#pragma unroll
  for (int j = 0; j < NT; ++j) xr[j] = xb + size_t(j < nt ? tok[j] : tok[0]) * rowb;
  float g0[NT], u0[NT], g1[NT], u1[NT];
#pragma unroll
  for (int j = 0; j < NT; ++j) g0[j] = u0[j] = g1[j] = u1[j] = 0.f;
  const int nch = int(rowb / 16);
#pragma unroll 2
  for (int c = lane; c < nch; c += 32) {
    const size_t ob = size_t(c) * 16;
    float fa[C::n], fb[C::n], fc[C::n], fd[C::n];
    C::cvt(ld_stream16(w1a + ob), fa);
    C::cvt(ld_stream16(w3a + ob), fb);
    C::cvt(ld_stream16(w1b + ob), fc);
    C::cvt(ld_stream16(w3b + ob), fd);
#pragma unroll
    for (int j = 0; j < NT; ++j) {
      if (j < nt) {
        float xv[C::n];
        C::cvt(ldg16(xr[j] + ob), xv);
#pragma unroll
        for (int i = 0; i < C::n; ++i) {
          g0[j] = fmaf(fa[i], xv[i], g0[j]);
          u0[j] = fmaf(fb[i], xv[i], u0[j]);
          g1[j] = fmaf(fc[i], xv[i], g1[j]);
          u1[j] = fmaf(fd[i], xv[i], u1[j]);
        }
      }
    }
  }
  float* h = reinterpret_cast<float*>(a.h);
#pragma unroll
  for (int j = 0; j < NT; ++j) {
    if (j < nt) {
      float ga = warp_sum(g0[j]), ua = warp_sum(u0[j]);
      float gb = warp_sum(g1[j]), ub = warp_sum(u1[j]);
      if (lane == j) {
        if (lblk) {  // LoRA: + s B1 (A1 x), + s B3 (A3 x)
          const LoraOffsets lo = lora_offsets(a.d, a.w, a.lrank);
          const float* u = a.u13 + size_t(q0 + j) * 2 * a.lrank;
          ga += lora_up<TW>(lblk, lo.b1, r0, u, a.lrank, a.lscale);
          gb += lora_up<TW>(lblk, lo.b1, r0 + 1, u, a.lrank, a.lscale);
          ua += lora_up<TW>(lblk, lo.b3, r0, u + a.lrank, a.lrank, a.lscale);
          ub += lora_up<TW>(lblk, lo.b3, r0 + 1, u + a.lrank, a.lrank, a.lscale);
        }
        float2 v = make_float2(silu(ga) * ua, silu(gb) * ub);
        *reinterpret_cast<float2*>(h + size_t(q0 + j) * a.w + r0) = v;
      }
    }
  }
}

// o[q, j] = W2[j] . h_q for output rows j = r0, r0 + 1 and NT permuted rows q0.. of a segment.
template <typename TW, int NT>
__device__ __forceinline__ void ffn2_tile(const FfnArgs& a, const char* blk, const void* lblk,
                                          int r0, int q0, int nt, int lane) {
  using C = W16<TW>;
  const size_t rowb = size_t(a.w) * sizeof(TW);
  const char* w2 = blk + size_t(2) * a.w * a.d * sizeof(TW);
  const char* wa = w2 + size_t(r0) * rowb;
  const char* wb = wa + rowb;
  const float* h = reinterpret_cast<const float*>(a.h);
  float s0[NT], s1[NT];
#pragma unroll
  for (int j = 0; j < NT; ++j) s0[j] = s1[j] = 0.f;
  const int nch = int(rowb / 16);
#pragma unroll 2
  for (int c = lane; c < nch; c += 32) {
    float fa[C::n], fb[C::n];
    C::cvt(ld_stream16(wa + size_t(c) * 16), fa);
    C::cvt(ld_stream16(wb + size_t(c) * 16), fb);
#pragma unroll
    for (int j = 0; j < NT; ++j) {
      if (j < nt) {
        const float4* hp = reinterpret_cast<const float4*>(h + size_t(q0 + j) * a.w + size_t(c) * C::n);
        float hv[C::n];
#pragma unroll
        for (int v = 0; v < C::n / 4; ++v) {
          const float4 t4 = hp[v];
          hv[4 * v] = t4.x; hv[4 * v + 1] = t4.y; hv[4 * v + 2] = t4.z; hv[4 * v + 3] = t4.w;
        }
#pragma unroll
        for (int i = 0; i < C::n; ++i) {
          s0[j] = fmaf(fa[i], hv[i], s0[j]);
          s1[j] = fmaf(fb[i], hv[i], s1[j]);
        }
      }
    }
  }
#pragma unroll
  for (int j = 0; j < NT; ++j) {
    if (j < nt) {
      float va = warp_sum(s0[j]), vb = warp_sum(s1[j]);
      if (lane == j) {
        if (lblk) {  // LoRA: + s B2 (A2 h)
          const size_t b2 = lora_offsets(a.d, a.w, a.lrank).b2;
          const float* u = a.u2 + size_t(q0 + j) * a.lrank;
          va += lora_up<TW>(lblk, b2, r0, u, a.lrank, a.lscale);
          vb += lora_up<TW>(lblk, b2, r0 + 1, u, a.lrank, a.lscale);
        }
        *reinterpret_cast<float2*>(a.o + size_t(q0 + j) * a.d + r0) = make_float2(va, vb);
      }
    }
  }
}

template <typename TW>
__global__ void __launch_bounds__(kWarps * 32) ffn13_kernel(const __grid_constant__ FfnArgs a) {
  pdl_wait();
  __shared__ Items it;
  build_items(it, a, a.w);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  for (int item = blockIdx.x; item < it.total; item += gridDim.x) {
    const int s = find_seg(it, item);
    const int r0 = (item - it.first[s]) * kRowsPerItem + warp * kRowsPerWarp;
    const char* blk = it.blk[s];
    const void* lblk = a.lrank ? a.lblk[s] : nullptr;
    const int q_begin = it.off[s], q_end = it.off[s + 1];
    for (int q0 = q_begin; q0 < q_end; q0 += kTokGroup) {
      const int nt = min(kTokGroup, q_end - q0);
      int tok[kTokGroup];
#pragma unroll
      for (int j = 0; j < kTokGroup; ++j) tok[j] = j < nt ? a.perm[q0 + j] : 0;
      if (nt == 1) ffn13_tile<TW, 1>(a, blk, lblk, r0, q0, nt, tok, lane);
      else if (nt == 2) ffn13_tile<TW, 2>(a, blk, lblk, r0, q0, nt, tok, lane);
      else if (nt <= 4) ffn13_tile<TW, 4>(a, blk, lblk, r0, q0, nt, tok, lane);
      else ffn13_tile<TW, 8>(a, blk, lblk, r0, q0, nt, tok, lane);
    }
  }
}

template <typename TW>
__global__ void __launch_bounds__(kWarps * 32) ffn2_kernel(const __grid_constant__ FfnArgs a) {
  pdl_wait();
  __shared__ Items it;
  build_items(it, a, a.d);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  for (int item = blockIdx.x; item < it.total; item += gridDim.x) {
    const int s = find_seg(it, item);
    const int r0 = (item - it.first[s]) * kRowsPerItem + warp * kRowsPerWarp;
    const char* blk = it.blk[s];
    const void* lblk = a.lrank ? a.lblk[s] : nullptr;
    const int q_begin = it.off[s], q_end = it.off[s + 1];
    for (int q0 = q_begin; q0 < q_end; q0 += kTokGroup) {
      const int nt = min(kTokGroup, q_end - q0);
      if (nt == 1) ffn2_tile<TW, 1>(a, blk, lblk, r0, q0, nt, lane);
      else if (nt == 2) ffn2_tile<TW, 2>(a, blk, lblk, r0, q0, nt, lane);
      else if (nt <= 4) ffn2_tile<TW, 4>(a, blk, lblk, r0, q0, nt, lane);
      else ffn2_tile<TW, 8>(a, blk, lblk, r0, q0, nt, lane);
    }
  }
}

// y[t] = sum_k g[t,k] o[pos(t,k)] + sum_s o[shared row s of t] (Section 3.1), every o row first
// summed over its partial planes in plane order, the rows in k order then shared order (a shared
// row enters as fma(1, v, acc), which is exactly acc + v). The loads are what take time: each
// thread takes its token's rows four at a time and issues the four index loads, then all 4 x KS
// plane loads, before adding anything, so a row group costs two round trips to L2 instead of one
// per row and plane. VEC outputs per thread: 4 (float4) while the planes are few, else 1 (more
// threads for the same outputs, and registers for 4 rows x KS planes).
template <typename TY, int KS, int VEC>
__global__ void __launch_bounds__(256) combine_kernel(const __grid_constant__ CombineArgs a) {
  using V = typename std::conditional<VEC == 4, float4, float>::type;
  pdl_wait();
  if (a.hdr->abort) return;
  const int nq = a.d / VEC;  // vectors per output row
  const int nr = a.K + a.S;
  const size_t total = size_t(a.T) * nq;
  for (size_t i = size_t(blockIdx.x) * blockDim.x + threadIdx.x; i < total;
       i += size_t(gridDim.x) * blockDim.x) {
    const int t = int(i / nq), c = int(i % nq) * VEC;
    float acc[VEC];
#pragma unroll
    for (int e = 0; e < VEC; ++e) acc[e] = 0.f;
    for (int r0 = 0; r0 < nr; r0 += 4) {
      size_t row[4];
      float g[4];
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const int r = r0 + j;
        row[j] = 0;
        g[j] = 1.f;
        if (r < a.K) {
          row[j] = size_t(a.pos[size_t(t) * a.K + r]);
          g[j] = a.gate[size_t(t) * a.K + r];
        } else if (r < nr) {
          row[j] = size_t(a.off[a.E + r - a.K] + t);
        }
      }
      V v[4][KS];
#pragma unroll
      for (int j = 0; j < 4; ++j)
        if (r0 + j < nr)
#pragma unroll
          for (int p = 0; p < KS; ++p)
            v[j][p] = *reinterpret_cast<const V*>(a.o + size_t(p) * a.o_plane + row[j] * a.d + c);
#pragma unroll
      for (int j = 0; j < 4; ++j)
        if (r0 + j < nr) {
          const float* f0 = reinterpret_cast<const float*>(&v[j][0]);
          float sum[VEC];
#pragma unroll
          for (int e = 0; e < VEC; ++e) sum[e] = f0[e];
#pragma unroll
          for (int p = 1; p < KS; ++p) {
            const float* f = reinterpret_cast<const float*>(&v[j][p]);
#pragma unroll
            for (int e = 0; e < VEC; ++e) sum[e] += f[e];
          }
#pragma unroll
          for (int e = 0; e < VEC; ++e) acc[e] = fmaf(g[j], sum[e], acc[e]);
        }
    }
    if constexpr (sizeof(TY) == 4) {
      float* y = reinterpret_cast<float*>(a.y) + size_t(t) * a.d + c;
#pragma unroll
      for (int e = 0; e < VEC; ++e) y[e] = acc[e];
    } else if constexpr (VEC == 4) {
      uint2 pk = make_uint2(pack2bf(acc[0], acc[1]), pack2bf(acc[2], acc[3]));
      *reinterpret_cast<uint2*>(reinterpret_cast<uint16_t*>(a.y) + size_t(t) * a.d + c) = pk;
    } else {
      reinterpret_cast<uint16_t*>(a.y)[size_t(t) * a.d + c] = f2bf(acc[0]);
    }
  }
}

int resident_blocks(const void* fn, int threads) {
  int nb = 1;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&nb, fn, threads, 0) != cudaSuccess || nb < 1) nb = 1;
  return nb;
}

template <typename TW>
cudaError_t launch_rowwise_typed(const FfnArgs& a, int num_sms, cudaStream_t s, int stages) {
  static int nb13 = resident_blocks(reinterpret_cast<const void*>(ffn13_kernel<TW>), kWarps * 32);
  static int nb2 = resident_blocks(reinterpret_cast<const void*>(ffn2_kernel<TW>), kWarps * 32);
  cudaError_t e = cudaSuccess;
  if (stages & 1) {
    prof_begin(kProfFfn13, s);
    e = launch_pdl(ffn13_kernel<TW>, dim3(num_sms * nb13), dim3(kWarps * 32), 0, s, a);
    prof_end(kProfFfn13, s);
    if (e == cudaSuccess) e = cudaGetLastError();
  }
  if (e != cudaSuccess || !(stages & 2)) return e;
  prof_begin(kProfFfn2, s);
  e = launch_pdl(ffn2_kernel<TW>, dim3(num_sms * nb2), dim3(kWarps * 32), 0, s, a);
  prof_end(kProfFfn2, s);
  return e != cudaSuccess ? e : cudaGetLastError();
}

template <typename TY, int KS, int VEC>
cudaError_t launch_combine_ks(const CombineArgs& a, cudaStream_t s) {
  const size_t total = size_t(a.T) * (a.d / VEC);
  size_t blocks = (total + 255) / 256;
  if (blocks > 4096) blocks = 4096;
  return launch_pdl(combine_kernel<TY, KS, VEC>, dim3(unsigned(blocks)), dim3(256), 0, s, a);
}

template <typename TY>
cudaError_t launch_combine_typed(const CombineArgs& a, cudaStream_t s) {
  switch (a.ks) {  // the contraction splits of the decode GEMM2 (decode_ksplit) and 1
    case 1: return launch_combine_ks<TY, 1, 4>(a, s);
    case 2: return launch_combine_ks<TY, 2, 4>(a, s);
    case 4: return launch_combine_ks<TY, 4, 1>(a, s);
    case 8: return launch_combine_ks<TY, 8, 1>(a, s);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace

cudaError_t launch_ffn_rowwise(const FfnArgs& a, int dtype, int num_sms, cudaStream_t s, int stages) {
  if (dtype != MCFT_F32) return cudaErrorInvalidValue;  // bf16 layers use the decode or TC path
  return launch_rowwise_typed<float>(a, num_sms, s, stages);
}

cudaError_t launch_combine(const CombineArgs& a, int dtype, cudaStream_t s) {
  if (a.T == 0) return cudaSuccess;
  prof_begin(kProfCombine, s);
  const cudaError_t e = dtype == MCFT_BF16 ? launch_combine_typed<uint16_t>(a, s)
                                           : launch_combine_typed<float>(a, s);
  prof_end(kProfCombine, s);
  return e != cudaSuccess ? e : cudaGetLastError();
}

}  // namespace mcft
