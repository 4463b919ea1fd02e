// Grouped expert GEMMs on the 5th-generation tensor cores (tcgen05 + TMEM), fed by TMA.
//
// Section 3.1: each routed expert is F(x) = W2 (silu(W1 x) * (W3 x)) (SwiGLU); with tokens
// permuted into per-expert segments (padded to 128 rows), the two expert GEMMs of a layer are
//   GEMM13: acc[m, 0:128] = xp[m] . W1[n0:n0+128]^T, acc[m, 128:256] = xp[m] . W3[n0:n0+128]^T,
//           h[m, n0:n0+128] = bf16(silu(acc_gate) * acc_up)             (fused epilogue)
//   GEMM2:  o[m, n0:n0+256] = h[m] . W2[n0:n0+256]^T                       (fp32 out)
// both D = A B^T with A and B K-major bf16, fp32 accumulators in tensor memory.
// With LoRA adapters (Section 3.2, Stage 2) every projection is W v + s B (A v). The down
// projections are skinny GEMMs on the same kernel (N = 16 or 32 columns, bf16 out, scaled by s):
//   DOWN13: U13[m] = s [A1 xp[m] | A3 xp[m]]    DOWN2: U2[m] = s A2 h[m]
// and the up projections ride on the expert GEMMs as one extra k-block per adapted tile,
// D += U B'^T, so the tensor cores add them to the accumulators and the epilogues are unchanged.
//
// One persistent CTA per SM, 6 warps (7 with adapters):
//   warp 0  - TMA producer (one thread): A tile 128x64 and B tile 256x64 per stage, 4 stages,
//             128-byte swizzle, one mbarrier with a transaction count per stage;
//   warp 1  - allocates 512 TMEM columns (two 128x256 fp32 accumulators) and issues
//             tcgen05.mma (M=128, N=256, K=16) from one thread; tcgen05.commit frees a stage /
//             publishes an accumulator;
//   warps 2-5 - epilogue: tcgen05.ld of their 32-lane quarter, SwiGLU or fp32, staged through
//             shared memory and stored as whole 128-byte row segments; they release the
//             accumulator so the next tile's MMAs overlap this tile's epilogue;
//   warp 6  - with adapters only: writes each adapted tile's extra k-block (see LoraOps).
// The down projections use the same roles with N = 16 or 32: 8 stages of 18-20 KB, 32 or 64 TMEM
// columns, bf16 rows written directly.
// Tiles are walked m-fastest inside groups of m-tiles so concurrently running CTAs share weight
// tiles (and the activation group) in L2. Every wait is bounded: after 2 s the kernel records
// MCFT_ERR_TIMEOUT, stops issuing, waits (bounded) for its copies and MMAs in flight, frees TMEM
// and returns.
#include <cuda.h>

#include "common.cuh"
#include "internal.h"
#include "mbar.cuh"

namespace mcft {
namespace {

constexpr int BM = 128, BN = 256, BK = 64;
constexpr int A_BYTES = BM * BK * 2;
constexpr int kMaxStages = 8;
constexpr int kThreads = 192;  // producer, MMA, 4 epilogue warps
constexpr int kBuilderWarp = 6;  // with adapters: one more warp writes the extra k-blocks
__host__ __device__ constexpr int threads_for(int lr) { return lr > 0 ? kThreads + 32 : kThreads; }

enum { EPI_SWIGLU = 0, EPI_F32 = 1, EPI_DOWN = 2 };

struct TcParams {
  CUtensorMap tma_a;
  CUtensorMap tma_b[kMaxSeg];
  const int* off;
  const WsHeader* hdr;
  void* out;
  unsigned* err;
  uint32_t wmask[3];  // segments that have weights
  int nseg, kblocks, ntiles_n, ldo, b_half, group_m;
  // LoRA (Stage 2): adapter block per segment (NULL: none); lug: the U operand rows (bf16;
  // GEMM13 [rows, 2r] = s [A1 x | A3 x], GEMM2 [rows, r] = s A2 h); lb0 / lb1: element offsets
  // of the up matrices (B1, B3 for GEMM13; B2 for GEMM2); lscale = s = alpha / r (DOWN scales
  // its output by it). b3d: the DOWN B map is 3-D ([A1; A3] planes) rather than 2-D (A2).
  const char* lblk[kMaxSeg];
  const uint16_t* lug;
  size_t lb0, lb1;
  float lscale;
  int b3d;
};

struct SmemCtl {
  uint64_t full[kMaxStages], empty[kMaxStages], tfull[2], tempty[2], drain;
  uint64_t bgo[2];  // with adapters: the producer hands the extra k-blocks' stages to the builder
  uint32_t tmem_base;
  int abort;
  int mt_total;
  int nseg;
  int off[kMaxSeg + 1];
};

// Geometry for an N-tile of NB columns: the expert GEMMs use NB = 256 (4 stages of 48 KB, two
// 128 x 256 fp32 accumulators = all 512 TMEM columns); the adapter down projection NB = 2r
// (8 stages of 18-20 KB, 32 or 64 TMEM columns).
// Epilogue store staging of the expert GEMMs: each epilogue warp writes 32 rows x 128 bytes of its
// output into shared memory (rows padded to 144 bytes: conflict-free 16-byte writes and reads),
// then stores them as whole 128-byte row segments, four rows per instruction.
constexpr int kOutRowBytes = 144;
constexpr int kOutWarpBytes = 32 * kOutRowBytes;
constexpr int kCtlBytes = (int(sizeof(SmemCtl)) + 15) / 16 * 16;

template <int NB>
struct Tile {
  static constexpr int B_BYTES = NB * BK * 2;
  static constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
  static constexpr int STAGES = NB >= 128 ? 4 : kMaxStages;
  static constexpr int TMEM_COLS = 2 * NB < 32 ? 32 : 2 * NB;
  // Instruction descriptor, kind::f16: D fp32 (bits 4-5 = 1), A bf16 (bits 7-9 = 1), B bf16
  // (bits 10-12 = 1), both K-major (bits 15, 16 = 0), N >> 3 at bit 17, M >> 4 at bit 24.
  static constexpr uint32_t IDESC = (1u << 4) | (1u << 7) | (1u << 10) |
                                    (uint32_t(NB >> 3) << 17) | (uint32_t(BM >> 4) << 24);
  static constexpr int OUT_STAGE = NB >= 128 ? 4 * kOutWarpBytes : 0;
  static constexpr int SMEM = STAGES * STAGE_BYTES + 1024 + kCtlBytes + OUT_STAGE;
  static_assert(NB % 16 == 0 && NB >= 16 && NB <= 256, "M = 128 needs N a multiple of 16");
  static_assert((TMEM_COLS & (TMEM_COLS - 1)) == 0 && TMEM_COLS <= 512, "TMEM allocation");
  static_assert(SMEM <= 227 * 1024, "shared memory");
};

__device__ __forceinline__ void tma_load_2d(uint32_t dst, const CUtensorMap* map, int c0, int c1,
                                            uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%2, %3}], [%4];" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(c0), "r"(c1), "r"(smem_u32(bar))
      : "memory");
}
__device__ __forceinline__ void tma_load_3d(uint32_t dst, const CUtensorMap* map, int c0, int c1,
                                            int c2, uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.tensor.3d.shared::cluster.global.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%2, %3, %4}], [%5];" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(c0), "r"(c1), "r"(c2), "r"(smem_u32(bar))
      : "memory");
}

__device__ __forceinline__ void tc_fence_before() {
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tc_fence_after() {
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}

// Shared-memory matrix descriptor, K-major, 128-byte swizzle: start address >> 4 (bits 0-13),
// leading byte offset (unused for this layout; 16 B), stride byte offset 1024 B between 8-row
// groups (bits 32-45), descriptor version 1 (bit 46), swizzle mode 2 = 128 B (bits 61-63).
__device__ __forceinline__ uint64_t sw128_desc(uint32_t saddr) {
  return uint64_t((saddr >> 4) & 0x3FFFu) | (uint64_t(1) << 16) | (uint64_t(1024 >> 4) << 32) |
         (uint64_t(1) << 46) | (uint64_t(2) << 61);
}

__device__ __forceinline__ void tc_mma(uint32_t d_tmem, uint64_t a, uint64_t b, uint32_t idesc,
                                       uint32_t acc) {
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
      " tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n}" ::"r"(d_tmem),
      "l"(a), "l"(b), "r"(idesc), "r"(acc)
      : "memory");
}

__device__ __forceinline__ void tc_commit(uint64_t* bar) {
  asm volatile(
      "tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
          smem_u32(bar))
      : "memory");
}

__device__ __forceinline__ void tmem_ld16(uint32_t taddr, uint32_t* r) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,"
      "%15}, [%16];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
        "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]),
        "=r"(r[14]), "=r"(r[15])
      : "r"(taddr));
}
__device__ __forceinline__ void tmem_ld_wait() {
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
}

// ---- CTA pairs (cta_group::2): one MMA of M = 256 over the shared memory of two CTAs ----
// Rank 0 of a 2-CTA cluster (the leader) issues the MMAs; each CTA holds 128 rows of A, 128 rows
// of B (its half of N) and its 128 accumulator rows in its own TMEM, at the same offsets.
__device__ __forceinline__ uint32_t cluster_rank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}
// Address of the same shared variable in cluster CTA `rank` (shared::cluster window).
__device__ __forceinline__ uint32_t peer_addr(const void* p, uint32_t rank) {
  uint32_t r;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(smem_u32(p)), "r"(rank));
  return r;
}
__device__ __forceinline__ void cluster_sync() {
  asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" :::
                   "memory");
}
__device__ __forceinline__ void mbar_arrive_cluster(uint32_t cluster_addr) {
  asm volatile("mbarrier.arrive.release.cluster.shared::cluster.b64 _, [%0];" ::"r"(cluster_addr)
               : "memory");
}
__device__ __forceinline__ bool mbar_try_wait_cl(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n .reg .pred p;\n mbarrier.try_wait.parity.acquire.cluster.shared::cta.b64 p, [%1], %2;\n"
      " selp.u32 %0, 1, 0, p;\n}"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}
// Bounded waits with cluster-scope acquire (the pair's barriers also complete from the peer CTA):
// false if the kernel is aborting or 2 s passed (then MCFT_ERR_TIMEOUT and the abort flag).
__device__ inline bool mbar_wait_cl(uint64_t* bar, uint32_t parity, volatile int* abort,
                                    unsigned* err) {
  if (mbar_try_wait_cl(bar, parity)) return true;
  const uint64_t t0 = globaltimer_ns();
  for (uint32_t i = 1;; ++i) {
    if (mbar_try_wait_cl(bar, parity)) return true;
    if ((i & 31) == 0) {
      if (*abort) return false;
      if (globaltimer_ns() - t0 > kTimeoutNs) {
        *abort = 1;
        set_error(err, kErrTimeout);
        return false;
      }
    }
  }
}
__device__ inline bool mbar_wait_drain_cl(uint64_t* bar, uint32_t parity, unsigned* err) {
  const uint64_t t0 = globaltimer_ns();
  while (!mbar_try_wait_cl(bar, parity)) {
    if (globaltimer_ns() - t0 > kTimeoutNs) {
      set_error(err, kErrTimeout);
      return false;
    }
  }
  return true;
}
// TMA tile load into this CTA's shared memory whose completion is counted on an mbarrier of
// either CTA of the pair (cluster address).
__device__ __forceinline__ void tma_load_2d_pair(uint32_t dst, const CUtensorMap* map, int c0,
                                                 int c1, uint32_t bar_cluster) {
  asm volatile(
      "cp.async.bulk.tensor.2d.cta_group::2.shared::cluster.global.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%2, %3}], [%4];" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(c0), "r"(c1), "r"(bar_cluster)
      : "memory");
}
__device__ __forceinline__ void tc_mma_pair(uint32_t d_tmem, uint64_t a, uint64_t b,
                                            uint32_t idesc, uint32_t acc) {
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
      " tcgen05.mma.cta_group::2.kind::f16 [%0], %1, %2, %3, p;\n}" ::"r"(d_tmem),
      "l"(a), "l"(b), "r"(idesc), "r"(acc)
      : "memory");
}
// Arrives on the mbarrier at this offset in both CTAs of the pair once the leader's MMAs issued
// so far have completed.
__device__ __forceinline__ void tc_commit_pair_both(uint64_t* bar) {
  asm volatile(
      "tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.multicast::cluster.b64"
      " [%0], %1;" ::"r"(smem_u32(bar)), "h"(static_cast<unsigned short>(3))
      : "memory");
}
__device__ __forceinline__ void tc_commit_pair(uint64_t* bar) {
  asm volatile(
      "tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
          smem_u32(bar))
      : "memory");
}

// Tile -> (m-tile, n-tile): groups of group_m m-tiles; inside a group, n-major then m.
__device__ __forceinline__ void tile_coords(int tile, int mt_total, int ntn, int G, int& mt,
                                            int& nt) {
  const int g = tile / (G * ntn);
  const int r = tile - g * G * ntn;
  const int gsz = min(G, mt_total - g * G);
  nt = r / gsz;
  mt = g * G + r % gsz;
}

__device__ __forceinline__ int seg_of_row(const SmemCtl* c, int row) {
  int s = 0;
  while (s + 1 < c->nseg && c->off[s + 1] <= row) ++s;
  return s;
}

// Whether an m-tile has work: always for the expert GEMMs; for the adapter down projection only
// when its segment (expert) has an adapter.
template <int EPI>
__device__ __forceinline__ bool tile_live(const SmemCtl* c, const TcParams& p, int mt) {
  if constexpr (EPI != EPI_DOWN) return true;
  const int s = seg_of_row(c, mt * BM);
  return ((p.wmask[s >> 5] >> (s & 31)) & 1u) != 0;
}

// The adapter operands of the extra k-block an adapted tile appends to its K loop (the up
// projections on the tensor cores): D += U B'^T with
//   GEMM13: U = [s A1 x | s A3 x] (K' = 2r), B' = [B1 rows | 0] for the gate half and
//           [0 | B3 rows] for the up half (block-diagonal, so one pass of N = 256 adds both);
//   GEMM2:  U = [s A2 h | 0], B' = [B2 rows | 0] (K' = r, zero-padded to 16).
// U and the B rows are bf16 in global memory (U written by the down-projection kernel / by
// GEMM13). The producer warp loads them into registers when it starts the tile, and writes them
// into the stage's A and B regions in the 128-byte-swizzled K-major layout the TMA tiles use
// (16-byte chunk c of row i at chunk c ^ (i % 8) of the row's 128 bytes) when the extra k-block's
// stage is free. Only the first K' columns of the stage are written and read.
template <int EPI, int LR>
struct LoraOps {
  static constexpr int KL = EPI == EPI_SWIGLU ? 2 * LR : (LR < 16 ? 16 : LR);  // K' of the block
  static constexpr int UC = (EPI == EPI_SWIGLU ? 2 * LR : LR) / 8;  // data chunks of a U row
  static constexpr int BC = LR / 8;                                 // data chunks of a B row
  static constexpr int CH = KL / 8;                                 // chunks written per row
  uint4 u[4][UC];  // tile rows 4 lane + i
  uint4 b[8][BC];  // B' rows lane + 32 i

  __device__ __forceinline__ void load(const TcParams& p, const char* lb, int mt, int nt,
                                       int lane) {
    const int ucols = EPI == EPI_SWIGLU ? 2 * LR : LR;
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const uint4* src =
          reinterpret_cast<const uint4*>(p.lug + (size_t(mt) * BM + 4 * lane + i) * ucols);
#pragma unroll
      for (int c = 0; c < UC; ++c) u[i][c] = __ldcg(src + c);
    }
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const int j = lane + 32 * i;
      size_t el;
      if constexpr (EPI == EPI_SWIGLU)
        el = j < BN / 2 ? p.lb0 + (size_t(nt) * (BN / 2) + j) * LR
                        : p.lb1 + (size_t(nt) * (BN / 2) + j - BN / 2) * LR;
      else
        el = p.lb0 + (size_t(nt) * BN + j) * LR;
      const uint4* src = reinterpret_cast<const uint4*>(lb + el * 2);
#pragma unroll
      for (int c = 0; c < BC; ++c) b[i][c] = __ldg(src + c);
    }
  }

  __device__ __forceinline__ void store(uint8_t* sa, uint8_t* sb, int lane) const {
    const uint4 z = make_uint4(0u, 0u, 0u, 0u);
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const int row = 4 * lane + i;
      uint4* dst = reinterpret_cast<uint4*>(sa + row * 128);
#pragma unroll
      for (int c = 0; c < CH; ++c) dst[c ^ (row & 7)] = c < UC ? u[i][c] : z;
    }
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const int row = lane + 32 * i;
      uint4* dst = reinterpret_cast<uint4*>(sb + row * 128);
      // GEMM13: gate rows hold B1 in chunks [0, BC), up rows B3 in chunks [BC, 2 BC)
      const int c0 = EPI == EPI_SWIGLU && row >= BN / 2 ? BC : 0;  // i >= 4: known when unrolled
#pragma unroll
      for (int c = 0; c < CH; ++c) {
        uint4 v = z;
#pragma unroll
        for (int e = 0; e < BC; ++e)
          if (c == c0 + e) v = b[i][e];
        dst[c ^ (row & 7)] = v;
      }
    }
  }
};

// Epilogue of one expert-GEMM tile for the 32 accumulator rows of an epilogue warp (TMEM lane
// quarter at taddr, output rows grow0 .. grow0 + 31, n-tile nt): SwiGLU to bf16 h (GEMM13) or fp32
// (GEMM2), staged through the warp's shared rows stg and stored as whole 128-byte row segments.
template <int EPI, int NB>
__device__ __forceinline__ void store_tile(const TcParams& p, uint8_t* stg, uint32_t taddr,
                                           size_t grow0, int nt, int lane) {
  if constexpr (EPI == EPI_SWIGLU) {
    // two rounds of 64 h columns (128 bytes of bf16 per row)
#pragma unroll 1
    for (int c0 = 0; c0 < NB / 2; c0 += 64) {
#pragma unroll
      for (int c = 0; c < 64; c += 16) {
        uint32_t g[16], u[16];
        tmem_ld16(taddr + c0 + c, g);
        tmem_ld16(taddr + NB / 2 + c0 + c, u);
        tmem_ld_wait();
        uint32_t pk[8];
#pragma unroll
        for (int i = 0; i < 8; ++i)
          pk[i] = pack2bf(silu(__uint_as_float(g[2 * i])) * __uint_as_float(u[2 * i]),
                          silu(__uint_as_float(g[2 * i + 1])) * __uint_as_float(u[2 * i + 1]));
        uint4* sw = reinterpret_cast<uint4*>(stg + lane * kOutRowBytes + c * 2);
        sw[0] = make_uint4(pk[0], pk[1], pk[2], pk[3]);
        sw[1] = make_uint4(pk[4], pk[5], pk[6], pk[7]);
      }
      __syncwarp();
      const size_t col = size_t(nt) * (NB / 2) + c0 + (lane & 7) * 8;
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        const int r = 4 * i + (lane >> 3);
        const uint4 v = *reinterpret_cast<const uint4*>(stg + r * kOutRowBytes + (lane & 7) * 16);
        *reinterpret_cast<uint4*>(reinterpret_cast<uint16_t*>(p.out) + (grow0 + r) * p.ldo + col) = v;
      }
      __syncwarp();
    }
  } else {
    // eight rounds of 32 fp32 columns (128 bytes per row)
#pragma unroll 1
    for (int c0 = 0; c0 < NB; c0 += 32) {
#pragma unroll
      for (int c = 0; c < 32; c += 16) {
        uint32_t v[16];
        tmem_ld16(taddr + c0 + c, v);
        tmem_ld_wait();
        uint4* sw = reinterpret_cast<uint4*>(stg + lane * kOutRowBytes + c * 4);
#pragma unroll
        for (int i = 0; i < 4; ++i) sw[i] = make_uint4(v[4 * i], v[4 * i + 1], v[4 * i + 2], v[4 * i + 3]);
      }
      __syncwarp();
      const size_t col = size_t(nt) * NB + c0 + (lane & 7) * 4;
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        const int r = 4 * i + (lane >> 3);
        const uint4 v = *reinterpret_cast<const uint4*>(stg + r * kOutRowBytes + (lane & 7) * 16);
        *reinterpret_cast<uint4*>(reinterpret_cast<float*>(p.out) + (grow0 + r) * p.ldo + col) = v;
      }
      __syncwarp();
    }
  }
}

template <int EPI, int LR, int NB>
__global__ void __launch_bounds__(threads_for(LR), 1) gemm_tc_kernel(const __grid_constant__ TcParams p) {
  using C = Tile<NB>;
  constexpr int STAGES = C::STAGES, STAGE_BYTES = C::STAGE_BYTES, TMEM_COLS = C::TMEM_COLS;
  constexpr int LRA = LR > 0 ? LR : 8;
  using LOps = LoraOps<EPI, LRA>;
  static_assert(LR == 0 || NB == BN, "adapters ride on the expert GEMMs");
  pdl_wait();
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = smem_u32(smem_raw);
  const uint32_t base = (raw + 1023u) & ~1023u;
  SmemCtl* ctl = reinterpret_cast<SmemCtl*>(smem_raw + (base - raw) + STAGES * STAGE_BYTES);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    int abort = p.hdr->abort;
    const int nseg = p.nseg;
    ctl->nseg = nseg;
    for (int s = 0; s <= nseg; ++s) ctl->off[s] = p.off[s];
    for (int s = 0; s < nseg && EPI != EPI_DOWN; ++s) {  // no adapter: no down projection
      if (ctl->off[s + 1] > ctl->off[s] && !((p.wmask[s >> 5] >> (s & 31)) & 1u)) {
        set_error(p.err, kErrInvalid);  // a selected expert without weights
        const_cast<WsHeader*>(p.hdr)->abort = 1;  // later kernels of the call skip their work
        abort = 1;
      }
    }
    ctl->abort = abort;
    ctl->mt_total = abort ? 0 : ctl->off[nseg] / BM;
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(&ctl->full[s], 1);
      mbar_init(&ctl->empty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&ctl->tfull[b], 1);
      mbar_init(&ctl->tempty[b], 4);
    }
    mbar_init(&ctl->drain, 1);
    mbar_init(&ctl->bgo[0], 1);
    mbar_init(&ctl->bgo[1], 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                     smem_u32(&ctl->tmem_base)),
                 "r"(TMEM_COLS)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();

  const uint32_t tmem = ctl->tmem_base;
  const int mt_total = ctl->mt_total;
  const int ntn = p.ntiles_n;
  const int tiles = mt_total * ntn;
  volatile int* abort = &ctl->abort;

  if (warp == 0) {
    // Producer: one thread issues the TMA copies. An adapted tile's extra k-block takes the next
    // stage after its K loop: the producer waits for that stage like any other and hands it to
    // the builder warp (bgo), which fills it. Every waiter thus waits on every phase of its
    // barriers in order, which a parity wait needs (it is ambiguous two phases away).
    if (lane == 0 && int(blockIdx.x) < tiles) {
      uint32_t it = 0, nl = 0;
      for (int tile = blockIdx.x; tile < tiles && !*abort; tile += gridDim.x) {
        int mt, nt;
        tile_coords(tile, mt_total, ntn, p.group_m, mt, nt);
        if (!tile_live<EPI>(ctl, p, mt)) continue;
        const int row0 = mt * BM;
        const int sg = seg_of_row(ctl, row0);
        const CUtensorMap* mb = &p.tma_b[sg];
        const int yb0 = EPI == EPI_SWIGLU ? nt * (NB / 2) : nt * NB;
        const int yb1 = EPI == EPI_SWIGLU ? p.b_half + nt * (NB / 2) : nt * NB + NB / 2;
        for (int kb = 0; kb < p.kblocks; ++kb, ++it) {
          const int s = int(it % STAGES);
          if (!mbar_wait(&ctl->empty[s], ((it / STAGES) & 1u) ^ 1u, abort, p.err)) break;
          const uint32_t sa = base + uint32_t(s) * STAGE_BYTES, sb = sa + A_BYTES;
          mbar_expect_tx(&ctl->full[s], STAGE_BYTES);
          tma_load_2d(sa, &p.tma_a, kb * BK, row0, &ctl->full[s]);
          if constexpr (EPI == EPI_DOWN) {
            if (p.b3d)  // [A1; A3]: one box of r rows x 2 planes
              tma_load_3d(sb, mb, kb * BK, 0, 0, &ctl->full[s]);
            else        // A2: a box of NB rows, those past r zero-filled
              tma_load_2d(sb, mb, kb * BK, 0, &ctl->full[s]);
          } else {
            tma_load_2d(sb, mb, kb * BK, yb0, &ctl->full[s]);
            tma_load_2d(sb + C::B_BYTES / 2, mb, kb * BK, yb1, &ctl->full[s]);
          }
        }
        if constexpr (LR > 0) {
          if (p.lblk[sg] != nullptr && !*abort) {  // the extra k-block's stage, for the builder
            const int s = int(it % STAGES);
            if (!mbar_wait(&ctl->empty[s], ((it / STAGES) & 1u) ^ 1u, abort, p.err)) break;
            mbar_arrive(&ctl->bgo[nl & 1u]);
            ++nl;
            ++it;
          }
        }
      }
      // Stages still in flight: the last STAGES issued ones (all consumed unless aborting).
      const uint32_t n_tail = it < STAGES ? it : STAGES;
      for (uint32_t j = it - n_tail; j < it; ++j)
        mbar_wait_drain(&ctl->full[j % STAGES], (j / STAGES) & 1u, p.err);
    }
  } else if (LR > 0 && warp == kBuilderWarp) {
    // Builder (adapters only): walks the producer's tile sequence and counts its stages; for the
    // n-th adapted tile it loads U and B' into registers when the tile starts, waits for the
    // producer's n-th hand-off (bgo[n % 2]: at most two are outstanding, since the MMAs stop at
    // the first unfilled stage and a tile has at least two TMA stages), writes the stage and
    // marks it full. Lane 0 waits; the outcome is broadcast.
    if (int(blockIdx.x) < tiles) {
      uint32_t it = 0, nl = 0;
      for (int tile = blockIdx.x; tile < tiles; tile += gridDim.x) {
        int mt, nt;
        tile_coords(tile, mt_total, ntn, p.group_m, mt, nt);
        const int sg = seg_of_row(ctl, mt * BM);
        it += uint32_t(p.kblocks);
        if (p.lblk[sg] == nullptr) continue;
        LOps lops;
        lops.load(p, p.lblk[sg], mt, nt, lane);
        int ok = 1;
        if (lane == 0) ok = mbar_wait(&ctl->bgo[nl & 1u], (nl >> 1) & 1u, abort, p.err);
        if (!__shfl_sync(0xffffffffu, ok, 0)) break;
        const int s = int(it % STAGES);
        const uint32_t sa = base + uint32_t(s) * STAGE_BYTES, sb = sa + A_BYTES;
        lops.store(smem_raw + (sa - raw), smem_raw + (sb - raw), lane);
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");  // for the MMA reads
        __syncwarp();
        if (lane == 0) mbar_arrive(&ctl->full[s]);
        ++nl;
        ++it;
      }
    }
  } else if (warp == 1) {
    if (lane == 0 && int(blockIdx.x) < tiles) {
      uint32_t it = 0, lt = 0;
      for (int tile = blockIdx.x; tile < tiles && !*abort; tile += gridDim.x) {
        bool lor = false;
        if constexpr (EPI == EPI_DOWN || LR > 0) {
          int mt, nt;
          tile_coords(tile, mt_total, ntn, p.group_m, mt, nt);
          if (!tile_live<EPI>(ctl, p, mt)) continue;
          if constexpr (LR > 0) lor = p.lblk[seg_of_row(ctl, mt * BM)] != nullptr;
        }
        const uint32_t b = lt & 1u;
        if (!mbar_wait(&ctl->tempty[b], ((lt >> 1) & 1u) ^ 1u, abort, p.err)) break;
        tc_fence_after();
        const uint32_t dt = tmem + b * NB;
        bool ok = true;
        const int nkb = p.kblocks + (lor ? 1 : 0);
        for (int kb = 0; kb < nkb; ++kb, ++it) {
          const int s = int(it % STAGES);
          if (!mbar_wait(&ctl->full[s], (it / STAGES) & 1u, abort, p.err)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t sa = base + uint32_t(s) * STAGE_BYTES, sb = sa + A_BYTES;
          const uint64_t da = sw128_desc(sa), db = sw128_desc(sb);
          if (LR == 0 || kb < p.kblocks) {
#pragma unroll
            for (int k = 0; k < BK / 16; ++k)  // +32 bytes along K per step inside the swizzle atom
              tc_mma(dt, da + uint64_t(2 * k), db + uint64_t(2 * k), C::IDESC,
                     (kb | k) != 0 ? 1u : 0u);
          } else {  // the adapters' up projections: D += U B'^T over K' columns
#pragma unroll
            for (int k = 0; k < LOps::KL / 16; ++k)
              tc_mma(dt, da + uint64_t(2 * k), db + uint64_t(2 * k), C::IDESC, 1u);
          }
          tc_commit(&ctl->empty[s]);
        }
        if (!ok) break;
        tc_commit(&ctl->tfull[b]);
        ++lt;
      }
      tc_commit(&ctl->drain);  // arrives once every MMA issued above has completed
      mbar_wait_drain(&ctl->drain, 0, p.err);
    }
  } else if (warp >= 2 && warp < 6) {
    const int q = warp & 3;  // TMEM lane quarter this warp may access
    const int row = q * 32 + lane;
    uint32_t lt = 0;
    for (int tile = blockIdx.x; tile < tiles; tile += gridDim.x) {
      int mt, nt;
      tile_coords(tile, mt_total, ntn, p.group_m, mt, nt);
      if (!tile_live<EPI>(ctl, p, mt)) continue;
      const uint32_t b = lt & 1u;
      int ok = 1;
      if (lane == 0) ok = mbar_wait(&ctl->tfull[b], (lt >> 1) & 1u, abort, p.err) ? 1 : 0;
      ok = __shfl_sync(0xffffffffu, ok, 0);
      if (!ok) break;
      tc_fence_after();
      const uint32_t taddr = tmem + b * NB + (uint32_t(q * 32) << 16);
      const size_t grow = size_t(mt) * BM + row;
      // this warp's staging rows; row r of the warp's quarter goes to global row grow0 + r
      uint8_t* stg = reinterpret_cast<uint8_t*>(ctl) + kCtlBytes + q * kOutWarpBytes;
      const size_t grow0 = size_t(mt) * BM + q * 32;
      if constexpr (EPI == EPI_DOWN) {  // U = s (A v) in bf16, the first ldo columns
        uint16_t* out = reinterpret_cast<uint16_t*>(p.out) + grow * p.ldo;
#pragma unroll
        for (int c = 0; c < NB; c += 16) {
          uint32_t v[16];
          tmem_ld16(taddr + c, v);
          tmem_ld_wait();
          uint32_t pk[8];
#pragma unroll
          for (int i = 0; i < 8; ++i)
            pk[i] = pack2bf(p.lscale * __uint_as_float(v[2 * i]),
                            p.lscale * __uint_as_float(v[2 * i + 1]));
          uint4* dst = reinterpret_cast<uint4*>(out + c);
          dst[0] = make_uint4(pk[0], pk[1], pk[2], pk[3]);
          if (c + 16 <= p.ldo) dst[1] = make_uint4(pk[4], pk[5], pk[6], pk[7]);
        }
      } else {
        store_tile<EPI, NB>(p, stg, taddr, grow0, nt, lane);
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&ctl->tempty[b]);
      ++lt;
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem),
                 "r"(TMEM_COLS)
                 : "memory");
  }
}

// The expert GEMMs on CTA pairs: tiles of 256 rows x 256 columns, one MMA of M = 256 per K step
// issued by the pair's leader over both CTAs' shared memory. Each CTA loads its 128 activation
// rows and its half of the tile's 256 weight rows (GEMM13: rank 0 the W1 rows, rank 1 the W3
// rows, i.e. the gate and up halves of N; GEMM2: 128 consecutive W2 rows each), so every weight
// element is read from shared memory once for the rows of both CTAs: a third less shared-memory
// traffic per MMA than the one-CTA tiles, and half the weight tiles fetched from L2 per tile row.
// Roles as in gemm_tc_kernel, 6 stages of 32 KB:
//   warp 0 (both CTAs) - TMA producer; the loads of both CTAs complete on the leader's full[s],
//             on which the leader expects the pair's bytes; each CTA waits on its own empty[s];
//   warp 1 - allocates the pair's TMEM (both CTAs); in the leader, issues the MMAs, whose commits
//             arrive on empty[s] and tfull[b] of both CTAs;
//   warps 2-5 (both CTAs) - epilogue of the CTA's 128 rows of the tile; they release the
//             accumulator on the leader's tempty[b] (eight arrivals: four warps per CTA).
// Segments are padded to 256 rows. Every wait is bounded. The leader drains its last stages'
// copies (both CTAs' bytes), the peer waits (bounded) until its last stages were consumed, and
// both CTAs leave through one cluster barrier after the leader's MMAs have completed, so neither
// exits while the other may still read its shared memory or arrive on its barriers.
constexpr int kPairRows = 2 * BM;
constexpr int kPairStages = 6;
constexpr int kPairStageBytes = A_BYTES + (BN / 2) * BK * 2;  // 128 activation + 128 weight rows
constexpr int kPairTmemCols = 2 * BN;                          // two 128 x 256 accumulators
constexpr uint32_t kPairIdesc = (1u << 4) | (1u << 7) | (1u << 10) | (uint32_t(BN >> 3) << 17) |
                                (uint32_t(kPairRows >> 4) << 24);
constexpr int kPairSmem = kPairStages * kPairStageBytes + 1024 + kCtlBytes + 4 * kOutWarpBytes;
static_assert(kPairSmem <= 227 * 1024, "shared memory");
static_assert(kPairStages <= kMaxStages, "stage barriers");

template <int EPI>
__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(kThreads, 1)
    gemm_tc_pair_kernel(const __grid_constant__ TcParams p) {
  pdl_wait();
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = smem_u32(smem_raw);
  const uint32_t base = (raw + 1023u) & ~1023u;  // the same offsets in both CTAs
  SmemCtl* ctl =
      reinterpret_cast<SmemCtl*>(smem_raw + (base - raw) + kPairStages * kPairStageBytes);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t rank = cluster_rank();
  const bool leader = rank == 0;

  if (threadIdx.x == 0) {
    // both CTAs find the same offsets and the same abort decision
    int abort = p.hdr->abort;
    const int nseg = p.nseg;
    ctl->nseg = nseg;
    for (int s = 0; s <= nseg; ++s) ctl->off[s] = p.off[s];
    for (int s = 0; s < nseg; ++s) {
      if (ctl->off[s + 1] > ctl->off[s] && !((p.wmask[s >> 5] >> (s & 31)) & 1u)) {
        set_error(p.err, kErrInvalid);  // a selected expert without weights
        const_cast<WsHeader*>(p.hdr)->abort = 1;
        abort = 1;
      }
    }
    ctl->abort = abort;
    ctl->mt_total = abort ? 0 : ctl->off[nseg] / kPairRows;
    for (int s = 0; s < kPairStages; ++s) {
      mbar_init(&ctl->full[s], 1);
      mbar_init(&ctl->empty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&ctl->tfull[b], 1);
      mbar_init(&ctl->tempty[b], 8);
    }
    mbar_init(&ctl->drain, 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                     smem_u32(&ctl->tmem_base)),
                 "r"(kPairTmemCols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;" ::: "memory");
  }
  tc_fence_before();
  cluster_sync();  // barriers initialised and TMEM allocated in both CTAs
  tc_fence_after();

  const uint32_t tmem = ctl->tmem_base;
  const int mt_total = ctl->mt_total;  // 256-row tiles
  const int ntn = p.ntiles_n;
  const int tiles = mt_total * ntn;
  const int cid = int(blockIdx.x >> 1), ncl = int(gridDim.x >> 1);  // pair, pairs
  volatile int* abort = &ctl->abort;

  if (warp == 0) {
    if (lane == 0 && cid < tiles) {
      uint32_t it = 0;
      for (int tile = cid; tile < tiles && !*abort; tile += ncl) {
        int mt, nt;
        tile_coords(tile, mt_total, ntn, p.group_m, mt, nt);
        const CUtensorMap* mb = &p.tma_b[seg_of_row(ctl, mt * kPairRows)];
        const int row0 = mt * kPairRows + int(rank) * BM;
        const int yb = EPI == EPI_SWIGLU ? int(rank) * p.b_half + nt * (BN / 2)
                                         : nt * BN + int(rank) * (BN / 2);
        for (int kb = 0; kb < p.kblocks; ++kb, ++it) {
          const int s = int(it % kPairStages);
          if (!mbar_wait_cl(&ctl->empty[s], ((it / kPairStages) & 1u) ^ 1u, abort, p.err)) break;
          const uint32_t sa = base + uint32_t(s) * kPairStageBytes, sb = sa + A_BYTES;
          const uint32_t fb = peer_addr(&ctl->full[s], 0);
          if (leader) mbar_expect_tx(&ctl->full[s], 2 * kPairStageBytes);
          tma_load_2d_pair(sa, &p.tma_a, kb * BK, row0, fb);
          tma_load_2d_pair(sb, mb, kb * BK, yb, fb);
        }
      }
      // Stages still in flight: the leader waits for their bytes (both CTAs'), the peer until
      // the leader's MMAs consumed them; after the first wait that runs out (an aborted pair,
      // 2 s: nothing is in flight any more) the rest are skipped.
      const uint32_t n_tail = it < kPairStages ? it : kPairStages;
      for (uint32_t j = it - n_tail; j < it; ++j) {
        uint64_t* bar = leader ? &ctl->full[j % kPairStages] : &ctl->empty[j % kPairStages];
        if (!mbar_wait_drain_cl(bar, (j / kPairStages) & 1u, p.err)) break;
      }
    }
  } else if (warp == 1) {
    if (leader && lane == 0 && cid < tiles) {
      uint32_t it = 0, lt = 0;
      for (int tile = cid; tile < tiles && !*abort; tile += ncl) {
        const uint32_t b = lt & 1u;
        if (!mbar_wait_cl(&ctl->tempty[b], ((lt >> 1) & 1u) ^ 1u, abort, p.err)) break;
        tc_fence_after();
        const uint32_t dt = tmem + b * BN;
        bool ok = true;
        for (int kb = 0; kb < p.kblocks; ++kb, ++it) {
          const int s = int(it % kPairStages);
          if (!mbar_wait_cl(&ctl->full[s], (it / kPairStages) & 1u, abort, p.err)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t sa = base + uint32_t(s) * kPairStageBytes, sb = sa + A_BYTES;
          const uint64_t da = sw128_desc(sa), db = sw128_desc(sb);
#pragma unroll
          for (int k = 0; k < BK / 16; ++k)
            tc_mma_pair(dt, da + uint64_t(2 * k), db + uint64_t(2 * k), kPairIdesc,
                        (kb | k) != 0 ? 1u : 0u);
          tc_commit_pair_both(&ctl->empty[s]);
        }
        if (!ok) break;
        tc_commit_pair_both(&ctl->tfull[b]);
        ++lt;
      }
      tc_commit_pair(&ctl->drain);  // arrives once every MMA issued above has completed
      mbar_wait_drain_cl(&ctl->drain, 0, p.err);
    }
  } else if (warp >= 2 && warp < 6) {
    const int q = warp & 3;  // TMEM lane quarter this warp may access
    uint8_t* stg = reinterpret_cast<uint8_t*>(ctl) + kCtlBytes + q * kOutWarpBytes;
    uint32_t lt = 0;
    for (int tile = cid; tile < tiles; tile += ncl) {
      int mt, nt;
      tile_coords(tile, mt_total, ntn, p.group_m, mt, nt);
      const uint32_t b = lt & 1u;
      int ok = 1;
      if (lane == 0) ok = mbar_wait_cl(&ctl->tfull[b], (lt >> 1) & 1u, abort, p.err) ? 1 : 0;
      ok = __shfl_sync(0xffffffffu, ok, 0);
      if (!ok) break;
      tc_fence_after();
      const uint32_t taddr = tmem + b * BN + (uint32_t(q * 32) << 16);
      const size_t grow0 = size_t(mt) * kPairRows + rank * BM + q * 32;
      store_tile<EPI, BN>(p, stg, taddr, grow0, nt, lane);
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive_cluster(peer_addr(&ctl->tempty[b], 0));
      ++lt;
    }
  }

  tc_fence_before();
  cluster_sync();  // the leader's MMAs drained, every copy landed, both epilogues done
  if (warp == 1) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, %1;" ::"r"(tmem),
                 "r"(kPairTmemCols)
                 : "memory");
  }
}

typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                   const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                   const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                   CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
  static EncodeTiledFn fn = [] {
    void* f = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &f, 12000, cudaEnableDefault,
                                         &q) != cudaSuccess ||
        q != cudaDriverEntryPointSuccess)
      f = nullptr;
    return reinterpret_cast<EncodeTiledFn>(f);
  }();
  return fn;
}

// bf16 matrix [rows, cols] row-major; box 64 columns (128 B, one swizzle span) x 128 rows.
bool encode_2d(CUtensorMap* m, const void* base, uint64_t cols, uint64_t rows) {
  EncodeTiledFn fn = encode_fn();
  if (!fn || (reinterpret_cast<uintptr_t>(base) & 15u) || ((cols * 2) & 15u)) return false;
  const cuuint64_t dims[2] = {cols, rows};
  const cuuint64_t strides[1] = {cols * 2};
  const cuuint32_t box[2] = {BK, 128};
  const cuuint32_t es[2] = {1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, es,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// The [A1; A3] rows of one adapter block as a 3-D map {d, r, 2}: plane 0 = A1 (element offset
// 0), plane 1 = A3 (plane stride a3 elements); box 64 columns x r rows x 2 planes, so one load
// fills the 2r rows of a down-projection B tile (A1 rows first), 128-byte swizzle.
bool encode_adapter_a13(CUtensorMap* m, const void* blk, uint64_t d, uint32_t r, uint64_t a3) {
  EncodeTiledFn fn = encode_fn();
  if (!fn || (reinterpret_cast<uintptr_t>(blk) & 15u) || ((d * 2) & 15u) || ((a3 * 2) & 15u))
    return false;
  const cuuint64_t dims[3] = {d, r, 2};
  const cuuint64_t strides[2] = {d * 2, a3 * 2};
  const cuuint32_t box[3] = {BK, r, 2};
  const cuuint32_t es[3] = {1, 1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(blk), dims, strides, box, es,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// A2 of one adapter block, [r, w] row-major, as a 2-D map with a box of 64 columns x 16 rows:
// for r = 8 the rows past r are outside the tensor and arrive as zeros (an N = 16 B tile).
bool encode_adapter_a2(CUtensorMap* m, const void* a2, uint64_t w, uint32_t r) {
  EncodeTiledFn fn = encode_fn();
  if (!fn || (reinterpret_cast<uintptr_t>(a2) & 15u) || ((w * 2) & 15u) || r > 16) return false;
  const cuuint64_t dims[2] = {w, r};
  const cuuint64_t strides[1] = {w * 2};
  const cuuint32_t box[2] = {BK, 16};
  const cuuint32_t es[2] = {1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(a2), dims, strides, box, es,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

constexpr size_t kSmallSegGroupMB = 2;  // group budget when routed experts have few m-tiles
// With CTA-pair tiles selected, layers whose routed experts average at least this many rows run
// on pairs (segments padded to 256 rows); with fewer the extra padding would dominate.
constexpr int kPairMinRows = 512;

int group_for(size_t a_tile_bytes, size_t budget_mb) {
  const size_t budget = budget_mb << 20;  // activation rows kept hot in L2 per group
  size_t g = budget / (a_tile_bytes ? a_tile_bytes : 1);
  return g < 1 ? 1 : int(g > 4096 ? 4096 : g);
}

template <int EPI, int LR, int NB>
cudaError_t launch_one(const TcParams& p, int grid, cudaStream_t s) {
  static cudaError_t attr = cudaFuncSetAttribute(
      gemm_tc_kernel<EPI, LR, NB>, cudaFuncAttributeMaxDynamicSharedMemorySize, Tile<NB>::SMEM);
  if (attr != cudaSuccess) return attr;
  const int kid = EPI == EPI_SWIGLU ? kProfGemm13 : EPI == EPI_F32 ? kProfGemm2 : kProfLora;
  prof_begin(kid, s);
  gemm_tc_kernel<EPI, LR, NB><<<grid, threads_for(LR), Tile<NB>::SMEM, s>>>(p);
  prof_end(kid, s);
  return cudaGetLastError();
}

// One pair per two SMs that can hold one at a time (one CTA per SM): a persistent grid of pairs
// that all run at once, so no pair's tiles wait for another pair to exit.
template <int EPI>
cudaError_t launch_pair(const TcParams& p, int num_sms, cudaStream_t s) {
  static cudaError_t attr = cudaFuncSetAttribute(
      gemm_tc_pair_kernel<EPI>, cudaFuncAttributeMaxDynamicSharedMemorySize, kPairSmem);
  if (attr != cudaSuccess) return attr;
  static const int pairs = [num_sms] {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(unsigned(num_sms & ~1));
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = kPairSmem;
    int n = 0;
    if (cudaOccupancyMaxActiveClusters(&n, gemm_tc_pair_kernel<EPI>, &cfg) != cudaSuccess) {
      (void)cudaGetLastError();
      n = 0;
    }
    return n;
  }();
  if (pairs < 1) return cudaErrorInvalidConfiguration;
  const int kid = EPI == EPI_SWIGLU ? kProfGemm13Pair : kProfGemm2Pair;
  prof_begin(kid, s);
  gemm_tc_pair_kernel<EPI><<<2 * pairs, kThreads, kPairSmem, s>>>(p);
  prof_end(kid, s);
  return cudaGetLastError();
}

template <int EPI>
cudaError_t launch_rank(const TcParams& p, int rank, int num_sms, cudaStream_t s) {
  switch (rank) {
    case 0: return launch_one<EPI, 0, BN>(p, num_sms, s);
    case 8: return launch_one<EPI, 8, BN>(p, num_sms, s);
    case 16: return launch_one<EPI, 16, BN>(p, num_sms, s);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace

bool tc_pair_tiles(int T, int K, int E, int lrank) {
  return lrank == 0 && size_t(T) * K >= size_t(kPairMinRows) * E;
}

cudaError_t launch_ffn_tc(const FfnArgs& a, const void* xp, int mcap, int pad, int num_sms,
                          cudaStream_t s, int stages) {
  const bool pair = pad == kPairRows;
  if (pair ? a.lrank != 0 : pad != BM) return cudaErrorInvalidValue;
  TcParams p13, p2;
  memset(&p13, 0, sizeof(p13));
  memset(&p2, 0, sizeof(p2));
  const size_t d = size_t(a.d), w = size_t(a.w);
  if (!encode_2d(&p13.tma_a, xp, d, size_t(mcap))) return cudaErrorInvalidValue;
  if (!encode_2d(&p2.tma_a, a.h, w, size_t(mcap))) return cudaErrorInvalidValue;
  for (int sgi = 0; sgi < a.nseg; ++sgi) {
    const char* blk = reinterpret_cast<const char*>(a.wblk[sgi]);
    if (!blk) continue;
    if (!encode_2d(&p13.tma_b[sgi], blk, d, 2 * w)) return cudaErrorInvalidValue;
    if (!encode_2d(&p2.tma_b[sgi], blk + 2 * w * d * 2, w, d)) return cudaErrorInvalidValue;
    p13.wmask[sgi >> 5] |= 1u << (sgi & 31);
  }
  p2.wmask[0] = p13.wmask[0];
  p2.wmask[1] = p13.wmask[1];
  p2.wmask[2] = p13.wmask[2];
  for (TcParams* q : {&p13, &p2}) {
    q->off = a.off;
    q->hdr = a.hdr;
    q->err = a.err;
    q->nseg = a.nseg;
  }
  p13.out = a.h;
  p13.kblocks = int(d / BK);
  p13.ntiles_n = int(w / (BN / 2));
  p13.ldo = int(w);
  p13.b_half = int(w);
  // L2 budgets per group of m-tiles, from same-box sweeps over the Mixtral- and
  // DeepSeek-V2-Lite-shaped T = 4096 layers: with several m-tiles per routed expert (Mixtral)
  // GEMM13 is best at 24 MB and GEMM2 at 12 MB; with fewer than four on average (DeepSeek-V2-Lite:
  // 64 experts) small groups of about one expert's rows win (GEMM13 0.55 -> 0.60 of peak)
  // routed rows T * K: the permuted rows less the shared experts' and the segment padding
  const size_t routed = size_t(mcap) - size_t(a.T) * (a.nseg - a.E) - size_t(a.nseg) * (pad - 1);
  const bool small_segs = routed < size_t(4) * BM * a.E;
  const size_t mb13 = small_segs ? kSmallSegGroupMB : 24, mb2 = small_segs ? kSmallSegGroupMB : 12;
  p13.group_m = group_for(size_t(pad) * d * 2, mb13);
  p2.out = a.o;
  p2.kblocks = int(w / BK);
  p2.ntiles_n = int(d / BN);
  p2.ldo = int(d);
  p2.b_half = 0;
  p2.group_m = group_for(size_t(pad) * w * 2, mb2);
  if (a.lrank > 0) {
    const LoraOffsets lo = lora_offsets(a.d, a.w, a.lrank);
    for (int sgi = 0; sgi < a.nseg; ++sgi) {
      p13.lblk[sgi] = reinterpret_cast<const char*>(a.lblk[sgi]);
      p2.lblk[sgi] = p13.lblk[sgi];
    }
    // U13 and U2 (bf16, from the down-projection launches) feed the extra k-blocks
    p13.lug = reinterpret_cast<const uint16_t*>(a.u13);
    p13.lb0 = lo.b1;
    p13.lb1 = lo.b3;
    p2.lug = reinterpret_cast<const uint16_t*>(a.u2);
    p2.lb0 = lo.b2;
  }
  cudaError_t e = cudaSuccess;
  if (stages & 1)
    e = pair ? launch_pair<EPI_SWIGLU>(p13, num_sms, s)
             : launch_rank<EPI_SWIGLU>(p13, a.lrank, num_sms, s);
  if (e != cudaSuccess || !(stages & 2)) return e;
  return pair ? launch_pair<EPI_F32>(p2, num_sms, s) : launch_rank<EPI_F32>(p2, a.lrank, num_sms, s);
}

cudaError_t launch_lora_down_tc(const FfnArgs& a, const void* xp, int mcap, int num_sms,
                                cudaStream_t s, int stage) {
  TcParams p;
  memset(&p, 0, sizeof(p));
  const size_t d = size_t(a.d), w = size_t(a.w);
  const int r = a.lrank;
  if (r != 8 && r != 16) return cudaErrorInvalidValue;
  const bool s13 = stage == 1;
  const size_t K = s13 ? d : w;
  if (!encode_2d(&p.tma_a, s13 ? xp : a.h, K, size_t(mcap))) return cudaErrorInvalidValue;
  const LoraOffsets lo = lora_offsets(a.d, a.w, r);
  for (int sgi = 0; sgi < a.nseg; ++sgi) {
    const char* blk = reinterpret_cast<const char*>(a.lblk[sgi]);
    if (!blk) continue;  // no adapter: the tile is skipped (its U rows are never read)
    const bool ok = s13 ? encode_adapter_a13(&p.tma_b[sgi], blk, d, uint32_t(r), lo.a3)
                        : encode_adapter_a2(&p.tma_b[sgi], blk + lo.a2 * 2, w, uint32_t(r));
    if (!ok) return cudaErrorInvalidValue;
    p.wmask[sgi >> 5] |= 1u << (sgi & 31);
  }
  p.off = a.off;
  p.hdr = a.hdr;
  p.err = a.err;
  p.nseg = a.nseg;
  p.b3d = s13 ? 1 : 0;
  p.out = const_cast<float*>(s13 ? a.u13 : a.u2);  // bf16 [rows, 2r] / [rows, r]
  p.lscale = a.lscale;
  p.kblocks = int(K / BK);
  p.ntiles_n = 1;
  p.ldo = s13 ? 2 * r : r;
  p.group_m = 1;
  const int mtiles = (mcap + BM - 1) / BM;
  const int grid = mtiles < num_sms ? (mtiles > 0 ? mtiles : 1) : num_sms;
  // N = 2r for [A1; A3]; 16 for A2 (r = 8: rows 8-15 of the box are zero)
  return s13 && r == 16 ? launch_one<EPI_DOWN, 0, 32>(p, grid, s)
                        : launch_one<EPI_DOWN, 0, 16>(p, grid, s);
}

}  // namespace mcft
