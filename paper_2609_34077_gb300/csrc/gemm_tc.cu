// Grouped expert GEMMs on the 5th-generation tensor cores (tcgen05 + TMEM), fed by TMA.
//
// Section 3.1: each routed expert is F(x) = W2 (silu(W1 x) * (W3 x)) (SwiGLU); with tokens
// permuted into per-expert segments (padded to 128 rows), the two expert GEMMs of a layer are
//   GEMM13: acc[m, 0:128] = xp[m] . W1[n0:n0+128]^T, acc[m, 128:256] = xp[m] . W3[n0:n0+128]^T,
//           h[m, n0:n0+128] = bf16(silu(acc_gate) * acc_up)             (fused epilogue)
//   GEMM2:  o[m, n0:n0+256] = h[m] . W2[n0:n0+256]^T                       (fp32 out)
// both D = A B^T with A and B K-major bf16, fp32 accumulators in tensor memory.
//
// One persistent CTA per SM, 6 warps:
//   warp 0  - TMA producer (one thread): A tile 128x64 and B tile 256x64 per stage, 4 stages,
//             128-byte swizzle, one mbarrier with a transaction count per stage;
//   warp 1  - allocates 512 TMEM columns (two 128x256 fp32 accumulators) and issues
//             tcgen05.mma (M=128, N=256, K=16) from one thread; tcgen05.commit frees a stage /
//             publishes an accumulator;
//   warps 2-5 - epilogue: tcgen05.ld of their 32-lane quarter, SwiGLU or fp32 store; they release
//             the accumulator so the next tile's MMAs overlap this tile's epilogue.
// Tiles are walked m-fastest inside groups of m-tiles so concurrently running CTAs share weight
// tiles (and the activation group) in L2. Every wait is bounded: after 2 s the kernel records
// MCFT_ERR_TIMEOUT, stops issuing, waits (bounded) for its copies and MMAs in flight, frees TMEM
// and returns.
#include <cuda.h>

#include "common.cuh"
#include "internal.h"

namespace mcft {
namespace {

constexpr int BM = 128, BN = 256, BK = 64, STAGES = 4;
constexpr int A_BYTES = BM * BK * 2;
constexpr int B_BYTES = BN * BK * 2;
constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
constexpr int TMEM_COLS = 2 * BN;
constexpr int kThreads = 192;
constexpr uint64_t kTimeoutNs = 2000000000ull;

enum { EPI_SWIGLU = 0, EPI_F32 = 1 };

// Instruction descriptor, kind::f16: D fp32 (bits 4-5 = 1), A bf16 (bits 7-9 = 1),
// B bf16 (bits 10-12 = 1), both K-major (bits 15, 16 = 0), N >> 3 at bit 17, M >> 4 at bit 24.
constexpr uint32_t kIdesc = (1u << 4) | (1u << 7) | (1u << 10) | (uint32_t(BN >> 3) << 17) |
                            (uint32_t(BM >> 4) << 24);

struct TcParams {
  CUtensorMap tma_a;
  CUtensorMap tma_b[kMaxSeg];
  const int* off;
  const WsHeader* hdr;
  void* out;
  unsigned* err;
  uint32_t wmask[3];  // segments that have weights
  int nseg, kblocks, ntiles_n, ldo, b_half, group_m;
  // LoRA (Stage 2): adapter block per segment (NULL: none), down-projections u [rows, ustride],
  // element offsets of the up matrices (B1, B3 for GEMM13; B2 for GEMM2), scale alpha / r.
  const char* lblk[kMaxSeg];
  const float* lu;
  int lustride;
  size_t lb0, lb1;
  float lscale;
};

// s * <u, B[row]> for rank R (B rows of R bf16 values, u in registers).
template <int R>
__device__ __forceinline__ float lora_dot(const char* blk, size_t b_off, int row, const float* u,
                                          float scale) {
  const uint4* b = reinterpret_cast<const uint4*>(blk + (b_off + size_t(row) * R) * 2);
  float acc = 0.f;
#pragma unroll
  for (int v = 0; v < R / 8; ++v) {
    float w8[8];
    unpack8(__ldg(b + v), w8);
#pragma unroll
    for (int i = 0; i < 8; ++i) acc = fmaf(u[8 * v + i], w8[i], acc);
  }
  return scale * acc;
}

struct SmemCtl {
  uint64_t full[STAGES], empty[STAGES], tfull[2], tempty[2], drain;
  uint32_t tmem_base;
  int abort;
  int mt_total;
  int nseg;
  int off[kMaxSeg + 1];
};

constexpr int kSmemBytes = STAGES * STAGE_BYTES + 1024 + int(sizeof(SmemCtl));

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count) : "memory");
}
__device__ __forceinline__ void mbar_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)),
               "r"(bytes)
               : "memory");
}
__device__ __forceinline__ void mbar_arrive(uint64_t* bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}
__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n"
      " selp.u32 %0, 1, 0, p;\n}"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}

// Wait for the phase of `parity` to complete; false if the kernel is aborting or 2 s passed.
__device__ bool mbar_wait(uint64_t* bar, uint32_t parity, volatile int* abort, unsigned* err) {
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = globaltimer_ns();
  for (uint32_t i = 1;; ++i) {
    if (mbar_try_wait(bar, parity)) return true;
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

// Bounded wait used while draining (ignores the abort flag).
__device__ void mbar_wait_drain(uint64_t* bar, uint32_t parity, unsigned* err) {
  const uint64_t t0 = globaltimer_ns();
  while (!mbar_try_wait(bar, parity)) {
    if (globaltimer_ns() - t0 > kTimeoutNs) {
      set_error(err, kErrTimeout);
      return;
    }
  }
}

__device__ __forceinline__ void tma_load_2d(uint32_t dst, const CUtensorMap* map, int c0, int c1,
                                            uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%2, %3}], [%4];" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(c0), "r"(c1), "r"(smem_u32(bar))
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

__device__ __forceinline__ void tc_mma(uint32_t d_tmem, uint64_t a, uint64_t b, uint32_t acc) {
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
      " tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n}" ::"r"(d_tmem),
      "l"(a), "l"(b), "r"(kIdesc), "r"(acc)
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

template <int EPI, int LR>
__global__ void __launch_bounds__(kThreads, 1) gemm_tc_kernel(const __grid_constant__ TcParams p) {
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
    for (int s = 0; s < nseg; ++s) {
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
    if (lane == 0 && int(blockIdx.x) < tiles) {
      uint32_t it = 0;
      for (int tile = blockIdx.x; tile < tiles && !*abort; tile += gridDim.x) {
        int mt, nt;
        tile_coords(tile, mt_total, ntn, p.group_m, mt, nt);
        const int row0 = mt * BM;
        const CUtensorMap* mb = &p.tma_b[seg_of_row(ctl, row0)];
        const int yb0 = EPI == EPI_SWIGLU ? nt * (BN / 2) : nt * BN;
        const int yb1 = EPI == EPI_SWIGLU ? p.b_half + nt * (BN / 2) : nt * BN + BN / 2;
        for (int kb = 0; kb < p.kblocks; ++kb, ++it) {
          const int s = int(it % STAGES);
          if (!mbar_wait(&ctl->empty[s], ((it / STAGES) & 1u) ^ 1u, abort, p.err)) break;
          const uint32_t sa = base + uint32_t(s) * STAGE_BYTES, sb = sa + A_BYTES;
          mbar_expect_tx(&ctl->full[s], STAGE_BYTES);
          tma_load_2d(sa, &p.tma_a, kb * BK, row0, &ctl->full[s]);
          tma_load_2d(sb, mb, kb * BK, yb0, &ctl->full[s]);
          tma_load_2d(sb + B_BYTES / 2, mb, kb * BK, yb1, &ctl->full[s]);
        }
      }
      // Copies still in flight: the last STAGES issued ones (all consumed unless aborting).
      const uint32_t n_tail = it < STAGES ? it : STAGES;
      for (uint32_t j = it - n_tail; j < it; ++j)
        mbar_wait_drain(&ctl->full[j % STAGES], (j / STAGES) & 1u, p.err);
    }
  } else if (warp == 1) {
    if (lane == 0 && int(blockIdx.x) < tiles) {
      uint32_t it = 0, lt = 0;
      for (int tile = blockIdx.x; tile < tiles && !*abort; tile += gridDim.x, ++lt) {
        const uint32_t b = lt & 1u;
        if (!mbar_wait(&ctl->tempty[b], ((lt >> 1) & 1u) ^ 1u, abort, p.err)) break;
        tc_fence_after();
        const uint32_t dt = tmem + b * BN;
        bool ok = true;
        for (int kb = 0; kb < p.kblocks; ++kb, ++it) {
          const int s = int(it % STAGES);
          if (!mbar_wait(&ctl->full[s], (it / STAGES) & 1u, abort, p.err)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t sa = base + uint32_t(s) * STAGE_BYTES, sb = sa + A_BYTES;
          const uint64_t da = sw128_desc(sa), db = sw128_desc(sb);
#pragma unroll
          for (int k = 0; k < BK / 16; ++k)  // +32 bytes along K per step inside the swizzle atom
            tc_mma(dt, da + uint64_t(2 * k), db + uint64_t(2 * k), (kb | k) != 0 ? 1u : 0u);
          tc_commit(&ctl->empty[s]);
        }
        if (!ok) break;
        tc_commit(&ctl->tfull[b]);
      }
      tc_commit(&ctl->drain);  // arrives once every MMA issued above has completed
      mbar_wait_drain(&ctl->drain, 0, p.err);
    }
  } else {
    const int q = warp & 3;  // TMEM lane quarter this warp may access
    const int row = q * 32 + lane;
    uint32_t lt = 0;
    for (int tile = blockIdx.x; tile < tiles; tile += gridDim.x, ++lt) {
      int mt, nt;
      tile_coords(tile, mt_total, ntn, p.group_m, mt, nt);
      const uint32_t b = lt & 1u;
      int ok = 1;
      if (lane == 0) ok = mbar_wait(&ctl->tfull[b], (lt >> 1) & 1u, abort, p.err) ? 1 : 0;
      ok = __shfl_sync(0xffffffffu, ok, 0);
      if (!ok) break;
      tc_fence_after();
      const uint32_t taddr = tmem + b * BN + (uint32_t(q * 32) << 16);
      const size_t grow = size_t(mt) * BM + row;
      // LoRA down-projections of this row (A1 x, A3 x) or (A2 h), kept in registers
      constexpr int LRA = LR > 0 ? LR : 1;
      float ua[LRA], ub[LRA];
      const char* lb = nullptr;
      if constexpr (LR > 0) {
        lb = p.lblk[seg_of_row(ctl, mt * BM)];
        if (lb) {
          const float* uq = p.lu + grow * p.lustride;
#pragma unroll
          for (int j = 0; j < LR; ++j) {
            ua[j] = uq[j];
            ub[j] = EPI == EPI_SWIGLU ? uq[LR + j] : 0.f;
          }
        }
      }
      if constexpr (EPI == EPI_SWIGLU) {
        uint16_t* out = reinterpret_cast<uint16_t*>(p.out) + grow * p.ldo + size_t(nt) * (BN / 2);
#pragma unroll 1
        for (int c = 0; c < BN / 2; c += 16) {
          uint32_t g[16], u[16];
          tmem_ld16(taddr + c, g);
          tmem_ld16(taddr + BN / 2 + c, u);
          tmem_ld_wait();
          float gf[16], uf[16];
#pragma unroll
          for (int i = 0; i < 16; ++i) {
            gf[i] = __uint_as_float(g[i]);
            uf[i] = __uint_as_float(u[i]);
          }
          if constexpr (LR > 0) {
            if (lb) {  // + s B1 (A1 x), + s B3 (A3 x)
              const int n0 = nt * (BN / 2) + c;
#pragma unroll
              for (int i = 0; i < 16; ++i) {
                gf[i] += lora_dot<LR>(lb, p.lb0, n0 + i, ua, p.lscale);
                uf[i] += lora_dot<LR>(lb, p.lb1, n0 + i, ub, p.lscale);
              }
            }
          }
          uint32_t pk[8];
#pragma unroll
          for (int i = 0; i < 8; ++i)
            pk[i] = pack2bf(silu(gf[2 * i]) * uf[2 * i], silu(gf[2 * i + 1]) * uf[2 * i + 1]);
          uint4* dst = reinterpret_cast<uint4*>(out + c);
          dst[0] = make_uint4(pk[0], pk[1], pk[2], pk[3]);
          dst[1] = make_uint4(pk[4], pk[5], pk[6], pk[7]);
        }
      } else {
        float* out = reinterpret_cast<float*>(p.out) + grow * p.ldo + size_t(nt) * BN;
#pragma unroll 1
        for (int c = 0; c < BN; c += 16) {
          uint32_t v[16];
          tmem_ld16(taddr + c, v);
          tmem_ld_wait();
          float f[16];
#pragma unroll
          for (int i = 0; i < 16; ++i) f[i] = __uint_as_float(v[i]);
          if constexpr (LR > 0) {
            if (lb) {  // + s B2 (A2 h)
#pragma unroll
              for (int i = 0; i < 16; ++i) f[i] += lora_dot<LR>(lb, p.lb0, nt * BN + c + i, ua, p.lscale);
            }
          }
          float4* dst = reinterpret_cast<float4*>(out + c);
#pragma unroll
          for (int i = 0; i < 4; ++i) dst[i] = make_float4(f[4 * i], f[4 * i + 1], f[4 * i + 2], f[4 * i + 3]);
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&ctl->tempty[b]);
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

int group_for(size_t a_tile_bytes) {
  const size_t budget = size_t(48) << 20;  // activation rows kept hot in L2 per group
  size_t g = budget / (a_tile_bytes ? a_tile_bytes : 1);
  return g < 1 ? 1 : int(g > 4096 ? 4096 : g);
}

template <int EPI, int LR>
cudaError_t launch_one(const TcParams& p, int num_sms, cudaStream_t s) {
  static cudaError_t attr = cudaFuncSetAttribute(
      gemm_tc_kernel<EPI, LR>, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemBytes);
  if (attr != cudaSuccess) return attr;
  const int kid = EPI == EPI_SWIGLU ? kProfGemm13 : kProfGemm2;
  prof_begin(kid, s);
  gemm_tc_kernel<EPI, LR><<<num_sms, kThreads, kSmemBytes, s>>>(p);
  prof_end(kid, s);
  return cudaGetLastError();
}

template <int EPI>
cudaError_t launch_rank(const TcParams& p, int rank, int num_sms, cudaStream_t s) {
  switch (rank) {
    case 0: return launch_one<EPI, 0>(p, num_sms, s);
    case 8: return launch_one<EPI, 8>(p, num_sms, s);
    case 16: return launch_one<EPI, 16>(p, num_sms, s);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace

cudaError_t launch_ffn_tc(const FfnArgs& a, const void* xp, int mcap, int num_sms, cudaStream_t s,
                          int stages) {
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
  p13.group_m = group_for(size_t(BM) * d * 2);
  p2.out = a.o;
  p2.kblocks = int(w / BK);
  p2.ntiles_n = int(d / BN);
  p2.ldo = int(d);
  p2.b_half = 0;
  p2.group_m = group_for(size_t(BM) * w * 2);
  if (a.lrank > 0) {
    const LoraOffsets lo = lora_offsets(a.d, a.w, a.lrank);
    for (int sgi = 0; sgi < a.nseg; ++sgi) {
      p13.lblk[sgi] = reinterpret_cast<const char*>(a.lblk[sgi]);
      p2.lblk[sgi] = p13.lblk[sgi];
    }
    p13.lu = a.u13;
    p13.lustride = 2 * a.lrank;
    p13.lb0 = lo.b1;
    p13.lb1 = lo.b3;
    p13.lscale = a.lscale;
    p2.lu = a.u2;
    p2.lustride = a.lrank;
    p2.lb0 = lo.b2;
    p2.lscale = a.lscale;
  }
  cudaError_t e = cudaSuccess;
  if (stages & 1) e = launch_rank<EPI_SWIGLU>(p13, a.lrank, num_sms, s);
  if (e != cudaSuccess || !(stages & 2)) return e;
  return launch_rank<EPI_F32>(p2, a.lrank, num_sms, s);
}

}  // namespace mcft
