// Chained decode stack (host runtime): one decode step of L masked MoE layers on the residual
// stream, with the cache's device-driven fetch and, optionally, prefetch of each next layer's
// predicted experts. Host code only; every step of the arithmetic runs in the library's kernels
// through the C ABI entry points, so a step issues no host synchronisation and can be captured in
// a CUDA graph.
//
// Per layer l of a step (Section 3.1 Eq. topk with the soft prior of Eq. inference; the residual
// stream and block-input RMSNorm of the paper's models, Section 4 and Table 4):
//   u_0 = RMSNorm_0(x_0)                                      (first layer only)
//   (idx_l, g_l) = route(u_l; router_l, pi_l);  cache step of layer l
//   with prefetch: predicted idx of layer l+1 = route(RMSNorm_{l+1}(x_l); router_{l+1}, pi_{l+1}),
//     prefetch event of layer l+1 (its loads stream in behind layer l's misses)
//   y_l = layer l on u_l with its cached experts (fetch overlapped with the hits' compute)
//   x_{l+1} = x_l + y_l;  u_{l+1} = RMSNorm_{l+1}(x_{l+1})
// At batch 1 each layer's steps before its expert FFN run as one fused prologue launch (an 8-CTA
// cluster, prologue.cu) and the forward skips its permutation; larger batches use the separate
// kernels above. Both make the same decisions.
#include <cuda_runtime.h>
#include <string.h>

#include <vector>

#include "internal.h"

struct mcft_stack {
  mcft_layer_desc desc{};
  int L = 0, T_max = 0, n_prefetch = 0, last_T = 0;
  float eps = 0.f;
  mcft_cache* cache = nullptr;
  std::vector<const void*> routers, gammas, shared;  // [L], [L], [L*S]
  std::vector<float> priors;                         // [L*E]
  void* u = nullptr;       // [T_max, d] layer dtype
  void* u_spec = nullptr;  // [T_max, d]
  void* y = nullptr;       // [T_max, d]
  int32_t* idx = nullptr;  // [L, T_max, K]
  float* gate = nullptr;   // [L, T_max, K]
  int32_t* pred = nullptr; // [L, T_max, K] (layer 0 unused)
  float* gate_pred = nullptr;  // [T_max, K] scratch
  void* ws = nullptr;
  size_t ws_bytes = 0;
};

namespace {

void stack_free(mcft_stack* s) {
  if (!s) return;
  cudaFree(s->u);
  cudaFree(s->u_spec);
  cudaFree(s->y);
  cudaFree(s->idx);
  cudaFree(s->gate);
  cudaFree(s->pred);
  cudaFree(s->gate_pred);
  cudaFree(s->ws);
  delete s;
}

mcft_status stack_fail(mcft_status st, const char* msg) { return mcft::set_error_message(st, msg); }

}  // namespace

extern "C" {

mcft_status mcft_stack_create(const mcft_layer_desc* desc, int L, const void* const* routers,
                              const float* priors, const void* const* gammas,
                              const void* const* shared, float eps, mcft_cache* cache,
                              int n_prefetch, int T_max, mcft_stack** out) {
  if (!out) return stack_fail(MCFT_ERR_INVALID, "out is NULL");
  *out = nullptr;
  if (!desc || !routers || !priors || !gammas || !cache)
    return stack_fail(MCFT_ERR_INVALID, "NULL argument");
  if (L < 1 || T_max < 1) return stack_fail(MCFT_ERR_INVALID, "L and T_max must be positive");
  // one workspace serves every batch size up to T_max (the layout depends on T)
  size_t need = 0;
  for (int T = 1; T <= T_max; ++T) {
    size_t n = 0;
    mcft_status st = mcft_moe_workspace_size(desc, T, &n);  // validates desc
    if (st != MCFT_OK) return st;
    if (n > need) need = n;
  }
  if (desc->dtype == MCFT_BF16 && T_max > 64)
    return stack_fail(MCFT_ERR_UNSUPPORTED, "the cached decode path takes at most 64 bf16 tokens");
  if (!(eps >= 0.f) || eps > 1.f) return stack_fail(MCFT_ERR_INVALID, "eps must be in [0, 1]");
  const int E = desc->E, S = desc->n_shared, K = desc->K, d = desc->d;
  if (S > 0 && !shared) return stack_fail(MCFT_ERR_INVALID, "shared is NULL");
  for (int l = 0; l < L; ++l)
    if (!routers[l] || !gammas[l]) return stack_fail(MCFT_ERR_INVALID, "NULL router or gamma");
  for (int i = 0; i < L * E; ++i)
    if (!(priors[i] > 0.f) || priors[i] > 3.0e38f)
      return stack_fail(MCFT_ERR_INVALID, "every prior entry must be positive and finite");
  mcft_stack* s = new mcft_stack();
  s->desc = *desc;
  s->L = L;
  s->T_max = T_max;
  s->n_prefetch = n_prefetch;
  s->eps = eps;
  s->cache = cache;
  s->routers.assign(routers, routers + L);
  s->gammas.assign(gammas, gammas + L);
  if (S > 0) s->shared.assign(shared, shared + size_t(L) * S);
  s->priors.assign(priors, priors + size_t(L) * E);
  const size_t esz = desc->dtype == MCFT_BF16 ? 2 : 4;
  const size_t act = size_t(T_max) * d * esz, ids = size_t(L) * T_max * K;
  cudaError_t e = cudaSuccess;
  if (e == cudaSuccess) e = cudaMalloc(&s->u, act);
  if (e == cudaSuccess) e = cudaMalloc(&s->u_spec, act);
  if (e == cudaSuccess) e = cudaMalloc(&s->y, act);
  if (e == cudaSuccess) e = cudaMalloc(&s->idx, ids * 4);
  if (e == cudaSuccess) e = cudaMalloc(&s->gate, ids * 4);
  if (e == cudaSuccess) e = cudaMalloc(&s->pred, ids * 4);
  if (e == cudaSuccess) e = cudaMalloc(&s->gate_pred, size_t(T_max) * K * 4);
  if (e == cudaSuccess) e = cudaMalloc(&s->ws, need);
  if (e == cudaSuccess) e = cudaMemset(s->pred, 0xff, ids * 4);
  if (e != cudaSuccess) {
    stack_free(s);
    return stack_fail(e == cudaErrorMemoryAllocation ? MCFT_ERR_OOM : MCFT_ERR_CUDA,
                      "stack buffer allocation failed");
  }
  s->ws_bytes = need;
  *out = s;
  return MCFT_OK;
}

mcft_status mcft_stack_step(mcft_stack* s, float* x, int T, mcft_stream_t compute,
                            mcft_stream_t copy) {
  mcft::NvtxRange nvtx_range("mcft_stack_step");
  if (!s || !x) return stack_fail(MCFT_ERR_INVALID, "NULL stack or x");
  if (T < 1 || T > s->T_max) return stack_fail(MCFT_ERR_INVALID, "T must be in [1, T_max]");
  const mcft_layer_desc* desc = &s->desc;
  const int L = s->L, E = desc->E, S = desc->n_shared, K = desc->K;
  const size_t plane = size_t(s->T_max) * K;
  mcft_status st;
  if (T == 1 && K <= mcft::kMaxK && mcft::prologue_supported(desc->d, E, T)) {
    // batch 1: one fused prologue launch per layer (stream update, norm, routing, cache step,
    // prediction and prefetch of the next layer, permutation), then the forward without its
    // permutation; the last layer's output is added by a final residual update
    for (int l = 0; l < L; ++l) {
      int32_t* idx = s->idx + l * plane;
      float* gate = s->gate + l * plane;
      const bool pf = s->n_prefetch > 0 && l + 1 < L;
      st = mcft::stack_prologue(desc, x, l == 0 ? nullptr : s->y, s->gammas[l],
                                pf ? s->gammas[l + 1] : nullptr, s->eps, s->u, s->routers[l],
                                s->priors.data() + size_t(l) * E, idx, gate,
                                pf ? s->routers[l + 1] : nullptr,
                                pf ? s->priors.data() + size_t(l + 1) * E : nullptr,
                                pf ? s->pred + (l + 1) * plane : nullptr, s->gate_pred, s->cache, l,
                                s->n_prefetch, s->ws, s->ws_bytes, compute);
      if (st != MCFT_OK) return st;
      st = mcft::forward_cached_impl(desc, s->u, T, idx, gate, s->cache, l,
                                     S > 0 ? s->shared.data() + size_t(l) * S : nullptr, s->y,
                                     s->ws, s->ws_bytes, compute, copy, true);
      if (st != MCFT_OK) return st;
    }
    st = mcft_residual_rmsnorm(desc, x, s->y, T, nullptr, s->eps, nullptr, compute);
    if (st != MCFT_OK) return st;
    s->last_T = T;
    return MCFT_OK;
  }
  st = mcft_residual_rmsnorm(desc, x, nullptr, T, s->gammas[0], s->eps, s->u, compute);
  if (st != MCFT_OK) return st;
  for (int l = 0; l < L; ++l) {
    int32_t* idx = s->idx + l * plane;
    float* gate = s->gate + l * plane;
    st = mcft_route(desc, s->u, T, s->routers[l], MCFT_ROUTE_SOFT_PRIOR, nullptr,
                    s->priors.data() + size_t(l) * E, idx, gate, compute);
    if (st != MCFT_OK) return st;
    st = mcft_cache_step(s->cache, l, idx, T, K, compute);
    if (st != MCFT_OK) return st;
    if (s->n_prefetch > 0 && l + 1 < L) {
      int32_t* pred = s->pred + (l + 1) * plane;
      st = mcft_residual_rmsnorm(desc, x, nullptr, T, s->gammas[l + 1], s->eps, s->u_spec, compute);
      if (st != MCFT_OK) return st;
      st = mcft_route(desc, s->u_spec, T, s->routers[l + 1], MCFT_ROUTE_SOFT_PRIOR, nullptr,
                      s->priors.data() + size_t(l + 1) * E, pred, s->gate_pred, compute);
      if (st != MCFT_OK) return st;
      st = mcft_cache_prefetch(s->cache, l + 1, pred, T, K, s->n_prefetch, compute);
      if (st != MCFT_OK) return st;
    }
    st = mcft_moe_forward_cached(desc, s->u, T, idx, gate, s->cache, l,
                                 S > 0 ? s->shared.data() + size_t(l) * S : nullptr, s->y, s->ws,
                                 s->ws_bytes, compute, copy);
    if (st != MCFT_OK) return st;
    st = mcft_residual_rmsnorm(desc, x, s->y, T, l + 1 < L ? s->gammas[l + 1] : nullptr, s->eps,
                               s->u, compute);
    if (st != MCFT_OK) return st;
  }
  s->last_T = T;
  return MCFT_OK;
}

mcft_status mcft_stack_routing(const mcft_stack* s, int layer, int32_t* idx, float* gate,
                               int32_t* idx_pred, mcft_stream_t stream) {
  if (!s) return stack_fail(MCFT_ERR_INVALID, "NULL stack");
  if (layer < 0 || layer >= s->L) return stack_fail(MCFT_ERR_INVALID, "layer out of range");
  const size_t n = size_t(s->last_T) * s->desc.K, off = size_t(layer) * s->T_max * s->desc.K;
  cudaError_t e = cudaSuccess;
  if (idx) e = cudaMemcpyAsync(idx, s->idx + off, n * 4, cudaMemcpyDeviceToHost, stream);
  if (e == cudaSuccess && gate)
    e = cudaMemcpyAsync(gate, s->gate + off, n * 4, cudaMemcpyDeviceToHost, stream);
  if (e == cudaSuccess && idx_pred)
    e = cudaMemcpyAsync(idx_pred, s->pred + off, n * 4, cudaMemcpyDeviceToHost, stream);
  if (e == cudaSuccess) e = cudaStreamSynchronize(stream);
  if (e != cudaSuccess) return stack_fail(MCFT_ERR_CUDA, cudaGetErrorString(e));
  return MCFT_OK;
}

void mcft_stack_destroy(mcft_stack* s) {
  if (!s) return;
  cudaDeviceSynchronize();
  stack_free(s);
}

}  // extern "C"
