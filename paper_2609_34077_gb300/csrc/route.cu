// Router GEMV + mask / prior + Top-K + gate softmax: one CTA per token at decode sizes, tiles of
// 16 tokens on the tensor cores at prefill sizes (route_tile_kernel, bf16).
//
// z = W x (Section 3.1); the score is z (plain Top-K, Eq. topk), z restricted to m_e = 1 (hard
// mask, Eq. stage1) or z_e + log pi_e (soft prior, Eq. inference: log(p_e pi_e) = z_e + log pi_e
// - logsumexp(z), the same order as p_e pi_e). The K best scores are taken largest first, equal
// scores to the lower expert index. Gates come from p = softmax(z): renormalised over the active
// set (Mixtral) or p_i itself (DeepSeek).
//
// Layout: one CTA of 16 warps per token. The E x d router is split into tasks (expert, contraction
// part): with E >= 16 each warp owns whole experts; with fewer experts each expert is split into up
// to 16 / E parts so every warp has work. A lane loads its part's chunks of x and of the expert
// row together, up to 8 chunks of 16 bytes in flight per lane and pass (one pass for d <= 4096 at
// these expert counts), so a decode token's router (64 KB Mixtral, 256 KB DeepSeek) is read in
// about one memory round trip instead of one per expert. Partial sums are reduced with shuffles
// and added in shared memory in a fixed order; warp 0 ranks (two experts per lane, shuffle
// arg-max) and writes idx / gate.
#include <cooperative_groups.h>

#include <type_traits>

#include "common.cuh"
#include "internal.h"
#include "route_warp.cuh"

namespace mcft {
namespace {

namespace cg = cooperative_groups;

constexpr int kWarps = 16;
constexpr int kRouteCluster = 4;  // CTAs per token for routers of many experts

template <typename TX>
struct Chunk;  // 16 bytes of a row: 8 bf16 or 4 fp32
template <>
struct Chunk<__nv_bfloat16> {
  static constexpr int n = 8;
  __device__ static void unpack(uint4 v, float* f) { unpack8(v, f); }
};
template <>
struct Chunk<float> {
  static constexpr int n = 4;
  __device__ static void unpack(uint4 v, float* f) {
    f[0] = __uint_as_float(v.x); f[1] = __uint_as_float(v.y);
    f[2] = __uint_as_float(v.z); f[3] = __uint_as_float(v.w);
  }
};

// Contraction parts per expert: the largest power of two p with E * p <= kWarps that divides the
// row's chunk count (the same on host and device).
__host__ __device__ inline int route_parts(int E, int nchunk) {
  int p = 1;
  while (2 * p * E <= kWarps && nchunk % (2 * p) == 0) p *= 2;
  return p;
}

// One warp: the logit part of token row xrow over chunks [0, per_part) of expert row wp (16-byte
// chunks, lane-strided, NCH chunks in flight per lane and pass, then a warp sum).
template <typename TX, int NCH>
__device__ __forceinline__ float router_dot(const char* xp, const char* wp, int per_part) {
  using C = Chunk<TX>;
  const int lane = threadIdx.x & 31;
  float acc = 0.f;
  for (int base = 0; base < per_part; base += 32 * NCH) {
    uint4 xv[NCH], wv[NCH];
#pragma unroll
    for (int i = 0; i < NCH; ++i) {
      const int c = base + i * 32 + lane;
      if (c < per_part) {
        xv[i] = ldg16(xp + size_t(c) * 16);
        wv[i] = ldg16(wp + size_t(c) * 16);
      }
    }
#pragma unroll
    for (int i = 0; i < NCH; ++i) {
      if (base + i * 32 + lane < per_part) {
        float xf[C::n], wf[C::n];
        C::unpack(xv[i], xf);
        C::unpack(wv[i], wf);
#pragma unroll
        for (int j = 0; j < C::n; ++j) acc = fmaf(xf[j], wf[j], acc);
      }
    }
  }
  return warp_sum(acc);
}

// NCH = 16-byte chunks a lane keeps in flight per task and pass (2, 4 or 8).
template <typename TX, int NCH>
__global__ void __launch_bounds__(kWarps * 32) route_kernel(const __grid_constant__ RouteArgs a) {
  pdl_wait();
  __shared__ float part[kMaxE][kWarps];
  __shared__ float zs[kMaxE];
  const int t = blockIdx.x;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int E = a.E, d = a.d;
  const int nchunk = d / Chunk<TX>::n;
  const int parts = route_parts(E, nchunk);
  const int per_part = nchunk / parts;

  const char* xrow = reinterpret_cast<const char*>(a.x) + size_t(t) * d * sizeof(TX);
  const char* wr = reinterpret_cast<const char*>(a.w_router);
  const size_t wrow = size_t(d) * sizeof(TX);
  for (int task = warp; task < E * parts; task += kWarps) {
    const int e = task / parts, pt = task % parts;
    const char* xp = xrow + size_t(pt) * per_part * 16;
    const char* wp = wr + e * wrow + size_t(pt) * per_part * 16;
    const float acc = router_dot<TX, NCH>(xp, wp, per_part);
    if (lane == 0) part[e][pt] = acc;
  }
  __syncthreads();
  if (warp != 0) return;
  for (int e = lane; e < E; e += 32) {
    float v = 0.f;
    for (int p = 0; p < parts; ++p) v += part[e][p];
    zs[e] = v;
  }
  __syncwarp();

  rank_and_gate_warp(a, zs, t);
}

// Routers of many experts (E >= 32, whole rows per task in route_kernel too): each token is one
// 4-CTA thread-block cluster, one expert per warp instead of E / 16 in series, each logit computed
// exactly as route_kernel computes it (router_dot over the whole row, then 0 + the logit, as its
// sum over one part), written into the leader CTA's shared memory over distributed shared memory;
// after one cluster barrier the leader's first warp ranks. The routing is bit-identical to
// route_kernel's in a quarter of the serial dot products.
template <typename TX, int NCH>
__global__ void __cluster_dims__(kRouteCluster, 1, 1) __launch_bounds__(kWarps * 32)
    route_cluster_kernel(const __grid_constant__ RouteArgs a) {
  pdl_wait();
  __shared__ float zs[kMaxE];
  cg::cluster_group cluster = cg::this_cluster();
  const int crank = int(cluster.block_rank());
  const int t = blockIdx.x / kRouteCluster;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int E = a.E, d = a.d;
  const int nchunk = d / Chunk<TX>::n;
  const char* xrow = reinterpret_cast<const char*>(a.x) + size_t(t) * d * sizeof(TX);
  const char* wr = reinterpret_cast<const char*>(a.w_router);
  const size_t wrow = size_t(d) * sizeof(TX);
  float* lead = cluster.map_shared_rank(&zs[0], 0);
  for (int e = crank * kWarps + warp; e < E; e += kRouteCluster * kWarps) {
    const float acc = router_dot<TX, NCH>(xrow, wr + e * wrow, nchunk);
    if (lane == 0) lead[e] = 0.f + acc;
  }
  cluster.sync();  // every logit is in the leader's shared memory
  if (crank != 0 || warp != 0) return;
  rank_and_gate_warp(a, zs, t);
}

// Prefill-sized bf16 calls (T > kRouteTileMinT): the router is a skinny GEMM z[T, E] = x W^T,
// bound by reading x once. A CTA of 8 warps takes up to 16 tokens; the logits come from mma.sync
// m16n8k16 (bf16 products, exact in fp32, fp32 accumulation). The tokens are spread evenly over
// two CTAs per SM (at most 16 per CTA, the MMA's rows; rows past a CTA's tokens read as zero), so
// no SM streams twice the rows of another. Warp w takes contraction
// slice w of 8 for all NTW 8-expert column tiles (NTW = ceil(E / 8) rounded up to a power of two;
// rows past E read as zero), U 32-element chunks per pass with every load of a pass issued before
// its MMAs, so a warp's chain of dependent memory round trips is (d / 256) / U passes long. A lane
// of quad position c loads 16 bytes (elements 8c..8c+7 of a chunk) of token rows g and g + 8 and
// of expert row g of each tile, and feeds words 0-1 to one MMA and words 2-3 to the next: the
// contraction order inside a chunk is permuted identically for x and W, so every product is
// formed exactly once. The 8 slices are summed in shared memory in slice order and each warp then
// ranks two tokens with the same warp function as the per-token kernel. The fp32 order differs
// from route_kernel's by rounding only (about 1e-7 relative), far inside the near-tie band of the
// routing contract.
constexpr int kTileTokens = 16;
constexpr int kTileWarps = 8;

template <int NTW, int U>
__global__ void __launch_bounds__(kTileWarps * 32, 2)
    route_tile_kernel(const __grid_constant__ RouteArgs a, int tpc) {
  pdl_wait();
  __shared__ float part[kTileWarps][kTileTokens][kMaxE + 1];
  __shared__ float zs[kTileTokens][kMaxE];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int g = lane >> 2, c = lane & 3;
  const int E = a.E, d = a.d;
  const int t0 = blockIdx.x * tpc, t1 = min(a.T, t0 + tpc);  // this CTA's tokens
  const size_t row = size_t(d) * 2;
  const int nch = d / 32;
  const int c0 = warp * nch / kTileWarps, c1 = (warp + 1) * nch / kTileWarps;
  const bool ok0 = t0 + g < t1, ok1 = t0 + g + 8 < t1;
  // rows past the last token or expert read a valid row and are zeroed before use
  const char* xa = static_cast<const char*>(a.x) + size_t(ok0 ? t0 + g : 0) * row + c * 16;
  const char* xb = static_cast<const char*>(a.x) + size_t(ok1 ? t0 + g + 8 : 0) * row + c * 16;
  const char* wr = static_cast<const char*>(a.w_router) + c * 16;
  float acc[NTW][4];
#pragma unroll
  for (int j = 0; j < NTW; ++j) acc[j][0] = acc[j][1] = acc[j][2] = acc[j][3] = 0.f;
  const uint4 zero = make_uint4(0, 0, 0, 0);
  auto wrow = [&](int j) { return wr + size_t(j * 8 + g < E ? j * 8 + g : 0) * row; };
  auto pass = [&](int ch, auto nchunks) {
    constexpr int n = decltype(nchunks)::value;
    uint4 va[n], vb[n], vw[n][NTW];
#pragma unroll
    for (int i = 0; i < n; ++i) {
      const size_t o = size_t(ch + i) * 64;
      va[i] = ldg16(xa + o);
      vb[i] = ldg16(xb + o);
#pragma unroll
      for (int j = 0; j < NTW; ++j) vw[i][j] = ldg16(wrow(j) + o);
    }
#pragma unroll
    for (int i = 0; i < n; ++i) {
      if (!ok0) va[i] = zero;
      if (!ok1) vb[i] = zero;
#pragma unroll
      for (int j = 0; j < NTW; ++j) {
        if (j * 8 + g >= E) vw[i][j] = zero;
        mma16816(acc[j], va[i].x, vb[i].x, va[i].y, vb[i].y, vw[i][j].x, vw[i][j].y);
        mma16816(acc[j], va[i].z, vb[i].z, va[i].w, vb[i].w, vw[i][j].z, vw[i][j].w);
      }
    }
  };
  int ch = c0;
  for (; ch + U <= c1; ch += U) pass(ch, std::integral_constant<int, U>{});
  for (; ch < c1; ++ch) pass(ch, std::integral_constant<int, 1>{});
  // C fragment of tile j: rows g and g + 8 (tokens), columns 2c and 2c + 1 (experts of the tile)
#pragma unroll
  for (int j = 0; j < NTW; ++j) {
    const int e0 = j * 8 + 2 * c;
    part[warp][g][e0] = acc[j][0];
    part[warp][g][e0 + 1] = acc[j][1];
    part[warp][g + 8][e0] = acc[j][2];
    part[warp][g + 8][e0 + 1] = acc[j][3];
  }
  __syncthreads();
  for (int i = threadIdx.x; i < kTileTokens * E; i += blockDim.x) {
    const int t = i / E, e = i % E;
    float v = part[0][t][e];
#pragma unroll
    for (int k = 1; k < kTileWarps; ++k) v += part[k][t][e];
    zs[t][e] = v;
  }
  __syncthreads();
  for (int t = warp; t < kTileTokens; t += kTileWarps)
    if (t0 + t < t1) rank_and_gate_warp(a, zs[t], t0 + t);
}

cudaError_t launch_route_tile(const RouteArgs& a, int num_sms, cudaStream_t s) {
  // tokens per CTA: the T tokens spread evenly over two CTAs per SM (at most 16, the MMA's rows)
  const int slots = 2 * num_sms;
  const int tpc = min(kTileTokens, max(1, (a.T + slots - 1) / slots));
  const dim3 grid((a.T + tpc - 1) / tpc), block(kTileWarps * 32);
  const int nt = (a.E + 7) / 8;
  // chunks per pass: about 24 16-byte loads in flight per lane
  if (nt == 1) return launch_pdl(route_tile_kernel<1, 8>, grid, block, 0, s, a, tpc);
  if (nt == 2) return launch_pdl(route_tile_kernel<2, 6>, grid, block, 0, s, a, tpc);
  if (nt <= 4) return launch_pdl(route_tile_kernel<4, 4>, grid, block, 0, s, a, tpc);
  return launch_pdl(route_tile_kernel<8, 2>, grid, block, 0, s, a, tpc);
}

template <typename TX>
cudaError_t launch_typed(const RouteArgs& a, cudaStream_t s) {
  const int nchunk = a.d / Chunk<TX>::n;
  const int per_lane = (nchunk / route_parts(a.E, nchunk) + 31) / 32;  // chunks per lane and task
  dim3 grid(a.T), block(kWarps * 32);
  prof_begin(kProfRoute, s);
  if (sizeof(TX) == 2 && a.T > kRouteTileMinT) {  // prefill-sized: tensor-core tiles of 16 tokens
    const cudaError_t e = launch_route_tile(a, num_sms(), s);
    prof_end(kProfRoute, s);
    return e != cudaSuccess ? e : cudaGetLastError();
  }
  if (a.E >= 2 * kWarps) {  // whole rows per task: one cluster per token
    const dim3 cgrid(a.T * kRouteCluster);
    const cudaError_t e =
        per_lane <= 2   ? launch_pdl(route_cluster_kernel<TX, 2>, cgrid, block, 0, s, a)
        : per_lane <= 4 ? launch_pdl(route_cluster_kernel<TX, 4>, cgrid, block, 0, s, a)
                        : launch_pdl(route_cluster_kernel<TX, 8>, cgrid, block, 0, s, a);
    prof_end(kProfRoute, s);
    return e != cudaSuccess ? e : cudaGetLastError();
  }
  const cudaError_t e =
      per_lane <= 2   ? launch_pdl(route_kernel<TX, 2>, grid, block, 0, s, a)
      : per_lane <= 4 ? launch_pdl(route_kernel<TX, 4>, grid, block, 0, s, a)
                      : launch_pdl(route_kernel<TX, 8>, grid, block, 0, s, a);  // long rows: passes
  prof_end(kProfRoute, s);
  return e != cudaSuccess ? e : cudaGetLastError();
}

}  // namespace

cudaError_t launch_route(const RouteArgs& a, int dtype, cudaStream_t s) {
  if (a.T == 0) return cudaSuccess;
  return dtype == MCFT_BF16 ? launch_typed<__nv_bfloat16>(a, s) : launch_typed<float>(a, s);
}

}  // namespace mcft
