// Stage-1 mask machinery (Section 3.2, Eq. stage1 and Eq. ste).
//
// mask_sample: pi = softmax(m~) per layer and E' experts drawn without replacement from pi, as the
//   Gumbel-top-k rule with caller-provided uniforms: key_e = log pi_e - log(-log u_e), the E'
//   largest keys (ties to the lower index) form the binary mask. One warp per layer, two experts
//   per lane, E' rounds of a shuffle arg-max.
// gate_grad: dL/dg_{t,k} = < dL/dy_t , F_{A_{t,k}}(x_t) >, the expert outputs F being the rows the
//   forward left in its workspace (summed over its partial planes). One warp per assignment.
// mask_grad: dL/dm_e = sum over tokens t with e in A_t of g_{t,e} (dg_{t,e} - sum_i g_{t,i} dg_{t,i})
//   for renormalised gates, g_{t,e} dg_{t,e} for plain gates (the gates of the active experts are
//   computed from p * m with m = 1 on A). One cluster of 8 CTAs: each CTA takes a contiguous
//   share of the tokens, each lane one token at a time (its K contributions computed once), and
//   the warp sums every expert's contributions with a butterfly; the warps' and then the CTAs'
//   partials are added in a fixed order (the leader reads the others' shared memory), so the sum
//   is deterministic. Then dL/dm~ = (diag(pi) - pi pi^T) dL/dm (straight-through estimator and
//   softmax Jacobian), optionally accumulated over several steps (the paper accumulates T steps
//   per update), in the same launch.
#include <cooperative_groups.h>

#include "common.cuh"
#include "internal.h"

namespace cg = cooperative_groups;

namespace mcft {
namespace {

__global__ void __launch_bounds__(32) mask_sample_kernel(const __grid_constant__ MaskSampleArgs a) {
  pdl_wait();
  const int l = blockIdx.x, lane = threadIdx.x, E = a.E;
  const float* mt = a.m_tilde + size_t(l) * E;
  const float* u = a.uniforms + size_t(l) * E;
  float v[2], key[2];
  bool ok[2];
  float mx = -INFINITY;
#pragma unroll
  for (int j = 0; j < 2; ++j) {
    const int e = lane + 32 * j;
    v[j] = e < E ? mt[e] : -INFINITY;
    mx = fmaxf(mx, v[j]);
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
  float se = 0.f;
#pragma unroll
  for (int j = 0; j < 2; ++j) se += lane + 32 * j < E ? expf(v[j] - mx) : 0.f;
  se = warp_sum(se);
  const float lse = logf(se);
  bool bad = false;
#pragma unroll
  for (int j = 0; j < 2; ++j) {
    const int e = lane + 32 * j;
    ok[j] = e < E;
    key[j] = -INFINITY;
    if (ok[j]) {
      const float lp = v[j] - mx - lse;  // log pi_e
      a.pi[size_t(l) * E + e] = expf(lp);
      const float ue = u[e];
      if (!(ue > 0.f && ue < 1.f)) {
        bad = true;
        ok[j] = false;
      } else {
        key[j] = lp - logf(-logf(ue));
      }
    }
  }
  if (__any_sync(0xffffffffu, bad) && lane == 0) set_error(a.err, kErrInvalid);
  bool taken[2] = {false, false};
  for (int r = 0; r < a.e_keep; ++r) {
    float bv = -INFINITY;
    int bi = 1 << 30;
#pragma unroll
    for (int j = 0; j < 2; ++j) {
      const int e = lane + 32 * j;
      if (ok[j] && !taken[j] && (key[j] > bv || (key[j] == bv && e < bi) || bi == (1 << 30))) {
        bv = key[j];
        bi = e;
      }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      const float v2 = __shfl_xor_sync(0xffffffffu, bv, o);
      const int i2 = __shfl_xor_sync(0xffffffffu, bi, o);
      if (v2 > bv || (v2 == bv && i2 < bi)) { bv = v2; bi = i2; }
    }
#pragma unroll
    for (int j = 0; j < 2; ++j)
      if (lane + 32 * j == bi) taken[j] = true;
  }
#pragma unroll
  for (int j = 0; j < 2; ++j) {
    const int e = lane + 32 * j;
    if (e < E) a.mask[size_t(l) * E + e] = taken[j] ? 1 : 0;
  }
}

// Four consecutive dL/dy values of a row (bf16 or fp32) as fp32.
template <typename TY>
__device__ __forceinline__ void load_dy4(const void* row, int c, float* dy) {
  if constexpr (sizeof(TY) == 2) {
    const uint2 v = *reinterpret_cast<const uint2*>(reinterpret_cast<const uint16_t*>(row) + c);
    dy[0] = bf16lo(v.x); dy[1] = bf16hi(v.x); dy[2] = bf16lo(v.y); dy[3] = bf16hi(v.y);
  } else {
    const float4 v = *reinterpret_cast<const float4*>(reinterpret_cast<const float*>(row) + c);
    dy[0] = v.x; dy[1] = v.y; dy[2] = v.z; dy[3] = v.w;
  }
}

template <typename TY>
__global__ void __launch_bounds__(256) gate_grad_kernel(const __grid_constant__ GateGradArgs a) {
  pdl_wait();
  if (a.hdr->abort) return;
  const int lane = threadIdx.x & 31;
  const int n = a.T * a.K;
  for (int i = blockIdx.x * 8 + (threadIdx.x >> 5); i < n; i += gridDim.x * 8) {
    const int t = i / a.K;
    const size_t row = size_t(a.pos[i]) * a.d;
    float acc = 0.f;
    const void* dyrow = sizeof(TY) == 2
        ? static_cast<const void*>(reinterpret_cast<const uint16_t*>(a.dy) + size_t(t) * a.d)
        : static_cast<const void*>(reinterpret_cast<const float*>(a.dy) + size_t(t) * a.d);
    if (a.ks == 1) {  // one plane (the tcgen05 path): 8 chunks in flight per lane, summed in order
      for (int c0 = lane * 4; c0 < a.d; c0 += 128 * 8) {
        float4 o[8];
        float dy[8][4];
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          const int c = c0 + 128 * j;
          if (c < a.d) {
            o[j] = __ldcs(reinterpret_cast<const float4*>(a.o + row + c));
            load_dy4<TY>(dyrow, c, dy[j]);
          }
        }
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          if (c0 + 128 * j < a.d) {
            acc = fmaf(dy[j][0], o[j].x, acc);
            acc = fmaf(dy[j][1], o[j].y, acc);
            acc = fmaf(dy[j][2], o[j].z, acc);
            acc = fmaf(dy[j][3], o[j].w, acc);
          }
        }
      }
    } else {
      for (int c = lane * 4; c < a.d; c += 128) {
        float4 o = *reinterpret_cast<const float4*>(a.o + row + c);
        for (int p = 1; p < a.ks; ++p) {
          const float4 u = *reinterpret_cast<const float4*>(a.o + size_t(p) * a.o_plane + row + c);
          o.x += u.x; o.y += u.y; o.z += u.z; o.w += u.w;
        }
        float dy[4];
        load_dy4<TY>(dyrow, c, dy);
        acc = fmaf(dy[0], o.x, acc);
        acc = fmaf(dy[1], o.y, acc);
        acc = fmaf(dy[2], o.z, acc);
        acc = fmaf(dy[3], o.w, acc);
      }
    }
    acc = warp_sum(acc);
    if (lane == 0) a.dgate[i] = acc;
  }
}

constexpr int kGradCluster = 8, kGradWarps = 16;

__global__ void __cluster_dims__(kGradCluster, 1, 1) __launch_bounds__(kGradWarps * 32)
    mask_grad_kernel(const __grid_constant__ MaskGradArgs a) {
  pdl_wait();
  __shared__ float wpart[kGradWarps][kMaxE];
  __shared__ float cpart[kMaxE];  // this CTA's share of dL/dm
  cg::cluster_group cluster = cg::this_cluster();
  const int crank = int(cluster.block_rank());
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int E = a.E, K = a.K, T = a.T;
  const int per = (T + kGradCluster - 1) / kGradCluster;
  const int t0 = crank * per, t1 = min(T, t0 + per);
  float acc0 = 0.f, acc1 = 0.f;  // this warp's sums for experts lane and lane + 32
  for (int base = t0 + warp * 32; base < t1; base += kGradWarps * 32) {
    const int t = base + lane;
    int ids[kMaxK];
    float c[kMaxK];
#pragma unroll
    for (int k = 0; k < kMaxK; ++k) {
      ids[k] = -1;
      c[k] = 0.f;
    }
    if (t < t1) {
      float inner = 0.f;  // sum_i g_{t,i} dL/dg_{t,i}
      for (int k = 0; k < K; ++k)
        inner = fmaf(a.gate[size_t(t) * K + k], a.dgate[size_t(t) * K + k], inner);
#pragma unroll
      for (int k = 0; k < kMaxK; ++k) {
        if (k < K) {
          const float g = a.gate[size_t(t) * K + k], dg = a.dgate[size_t(t) * K + k];
          ids[k] = a.idx[size_t(t) * K + k];
          c[k] = a.gate_mode == MCFT_GATE_RENORM ? g * (dg - inner) : g * dg;
        }
      }
    }
    for (int e = 0; e < E; ++e) {
      float v = 0.f;
      bool has = false;
#pragma unroll
      for (int k = 0; k < kMaxK; ++k) {
        if (ids[k] == e) {
          v += c[k];
          has = true;
        }
      }
      if (!__any_sync(0xffffffffu, has)) continue;  // no token of this group picked e
      v = warp_sum(v);
      if (lane == (e & 31)) {
        if (e < 32) acc0 += v;
        else acc1 += v;
      }
    }
  }
  wpart[warp][lane] = acc0;
  wpart[warp][lane + 32] = acc1;
  __syncthreads();
  if (threadIdx.x < E) {
    float sum = 0.f;
    for (int w = 0; w < kGradWarps; ++w) sum += wpart[w][threadIdx.x];
    cpart[threadIdx.x] = sum;
  }
  cluster.sync();  // every CTA's share is in its shared memory
  if (crank == 0 && warp == 0) {
    float dm[2] = {0.f, 0.f};
    for (int r = 0; r < kGradCluster; ++r) {
      const float* pr = cluster.map_shared_rank(&cpart[0], r);
#pragma unroll
      for (int j = 0; j < 2; ++j)
        if (lane + 32 * j < E) dm[j] += pr[lane + 32 * j];
    }
    float sp = 0.f;  // pi . dL/dm
#pragma unroll
    for (int j = 0; j < 2; ++j) {
      const int e = lane + 32 * j;
      if (e < E) {
        a.dm[e] = dm[j];
        sp += a.pi[e] * dm[j];
      }
    }
    sp = warp_sum(sp);
#pragma unroll
    for (int j = 0; j < 2; ++j) {
      const int e = lane + 32 * j;
      if (e < E) {
        const float v = a.pi[e] * (dm[j] - sp);
        a.dm_tilde[e] = a.accumulate ? a.dm_tilde[e] + v : v;
      }
    }
  }
  cluster.sync();  // the leader has read the other CTAs' shared memory
}

}  // namespace

cudaError_t launch_mask_sample(const MaskSampleArgs& a, cudaStream_t s) {
  mask_sample_kernel<<<a.L, 32, 0, s>>>(a);
  return cudaGetLastError();
}

cudaError_t launch_gate_grad(const GateGradArgs& a, int dtype, cudaStream_t s) {
  const int n = a.T * a.K;
  int blocks = (n + 7) / 8;
  if (blocks > 4096) blocks = 4096;
  if (dtype == MCFT_BF16) gate_grad_kernel<uint16_t><<<blocks, 256, 0, s>>>(a);
  else gate_grad_kernel<float><<<blocks, 256, 0, s>>>(a);
  return cudaGetLastError();
}

cudaError_t launch_mask_grad(const MaskGradArgs& a, cudaStream_t s) {
  mask_grad_kernel<<<kGradCluster, kGradWarps * 32, 0, s>>>(a);
  return cudaGetLastError();
}

}  // namespace mcft
