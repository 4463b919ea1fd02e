// C ABI of libmcft (include/mcft.h): argument validation, workspace layout, kernel launches,
// the expert cache object and its fetch engine (one host-to-device copy per miss on a copy stream,
// ordered against the compute stream with events).
#include <cuda_runtime.h>
#include <stdarg.h>
#include <stdio.h>
#include <string.h>

#include <atomic>
#include <mutex>
#include <string>
#include <vector>

#include "common.cuh"
#include "internal.h"

namespace mcft {
namespace {

thread_local std::string g_last_error;

mcft_status fail(mcft_status st, const char* fmt, ...) __attribute__((format(printf, 2, 3)));
mcft_status fail(mcft_status st, const char* fmt, ...) {
  char buf[512];
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(buf, sizeof(buf), fmt, ap);
  va_end(ap);
  g_last_error = buf;
  return st;
}

mcft_status cuda_fail(cudaError_t e, const char* where) {
  return fail(e == cudaErrorMemoryAllocation ? MCFT_ERR_OOM : MCFT_ERR_CUDA, "%s: %s", where,
              cudaGetErrorString(e));
}

#define MCFT_CUDA(call)                                   \
  do {                                                    \
    cudaError_t e_ = (call);                              \
    if (e_ != cudaSuccess) return cuda_fail(e_, #call);   \
  } while (0)

__device__ unsigned g_device_error;  // one per device that loads the library

// Test hooks (mcft_test_inject): how many of the next pinned host allocations and host-driven
// expert copies fail as if the runtime had refused them, the decode FFN's wait limit, and whether
// the decode FFN withholds its GEMM13 items. All zero (off) unless a test sets them.
std::atomic<int> g_inject_pinned{0}, g_inject_copy{0}, g_inject_withhold{0};
// Expert-GEMM tile shape (mcft_set_tc_tiles): MCFT_TC_TILES_ONE_CTA unless set.
std::atomic<int> g_tc_tiles{MCFT_TC_TILES_ONE_CTA};
std::atomic<unsigned long long> g_inject_wait_ns{0};

// Consume one injected failure from counter n: true while it is positive.
bool take_injected(std::atomic<int>& n) {
  int v = n.load();
  while (v > 0)
    if (n.compare_exchange_weak(v, v - 1)) return true;
  return false;
}

cudaError_t host_alloc_mapped(void** p, size_t bytes) {
  if (take_injected(g_inject_pinned)) return cudaErrorMemoryAllocation;
  return cudaHostAlloc(p, bytes, cudaHostAllocMapped);
}

cudaError_t expert_copy(void* dst, const void* src, size_t bytes, cudaStream_t s) {
  if (take_injected(g_inject_copy)) return cudaErrorUnknown;
  return cudaMemcpyAsync(dst, src, bytes, cudaMemcpyHostToDevice, s);
}

}  // namespace

unsigned long long test_wait_limit_ns() {
  const unsigned long long v = g_inject_wait_ns.load();
  return v ? v : 2000000000ull;
}

bool test_withhold_gemm13() { return g_inject_withhold.load() != 0; }

namespace {

constexpr int kMaxDevices = 64;

int current_device() {
  int dev = 0;
  cudaGetDevice(&dev);
  return dev;
}

}  // namespace

int num_sms() {
  static int cache[kMaxDevices] = {0};
  const int dev = current_device();
  if (dev < kMaxDevices && cache[dev]) return cache[dev];
  int n = 0;
  cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
  if (n <= 0) n = 1;
  if (dev < kMaxDevices) cache[dev] = n;
  return n;
}

namespace {

size_t align256(size_t v) { return (v + 255) & ~size_t(255); }

// CTAs of the device-driven fetch kernel: a quarter of the SMs (the host link is the bound, and
// the rest of the GPU stays with the FFN of the experts that were hits).
int fetch_blocks() { return num_sms() / 4 > 0 ? num_sms() / 4 : 1; }

mcft_status check_desc(const mcft_layer_desc* d) {
  if (!d) return fail(MCFT_ERR_INVALID, "desc is NULL");
  if (d->d <= 0 || d->d % 64) return fail(MCFT_ERR_INVALID, "d = %d must be a positive multiple of 64", d->d);
  if (d->w <= 0 || d->w % 64) return fail(MCFT_ERR_INVALID, "w = %d must be a positive multiple of 64", d->w);
  if (d->E <= 0) return fail(MCFT_ERR_INVALID, "E = %d must be positive", d->E);
  if (d->K <= 0 || d->K > d->E) return fail(MCFT_ERR_INVALID, "K = %d must be in [1, E = %d]", d->K, d->E);
  if (d->E > kMaxE) return fail(MCFT_ERR_UNSUPPORTED, "E = %d > %d", d->E, kMaxE);
  if (d->K > kMaxK) return fail(MCFT_ERR_UNSUPPORTED, "K = %d > %d", d->K, kMaxK);
  if (d->n_shared < 0) return fail(MCFT_ERR_INVALID, "n_shared = %d < 0", d->n_shared);
  if (d->n_shared > kMaxShared) return fail(MCFT_ERR_UNSUPPORTED, "n_shared = %d > %d", d->n_shared, kMaxShared);
  if (d->gate != MCFT_GATE_RENORM && d->gate != MCFT_GATE_PLAIN)
    return fail(MCFT_ERR_INVALID, "unknown gate mode %d", d->gate);
  if (d->dtype != MCFT_F32 && d->dtype != MCFT_BF16)
    return fail(MCFT_ERR_INVALID, "unknown dtype %d", d->dtype);
  return MCFT_OK;
}

}  // namespace

mcft_status set_error_message(mcft_status st, const char* msg) { return fail(st, "%s", msg); }

unsigned* device_error_word() {
  static unsigned* cache[kMaxDevices] = {nullptr};
  static std::mutex mu;
  const int dev = current_device();
  std::lock_guard<std::mutex> lock(mu);
  if (dev < kMaxDevices && cache[dev]) return cache[dev];
  void* p = nullptr;
  if (cudaGetSymbolAddress(&p, g_device_error) != cudaSuccess) return nullptr;
  if (dev < kMaxDevices) cache[dev] = static_cast<unsigned*>(p);
  return static_cast<unsigned*>(p);
}

WsLayout ws_layout(int d, int E, int K, int w, int S, int dtype, int T, int lrank) {
  WsLayout L{};
  L.lrank = lrank;
  L.tc = dtype == MCFT_BF16 && T > 64 && d % 256 == 0 && w % 128 == 0;
  L.decode = !L.tc && dtype == MCFT_BF16;
  L.ks = L.decode ? decode_ksplit(T) : 1;
  L.pad = !L.tc ? 1
          : g_tc_tiles.load() == MCFT_TC_TILES_CTA_PAIR && tc_pair_tiles(T, K, E, lrank) ? 256
                                                                                       : 128;
  const int nseg = E + S;
  L.mcap = T * K + S * T + (L.tc ? nseg * (L.pad - 1) : 0);
  size_t o = 0;
  L.hdr = o;  o = align256(o + sizeof(WsHeader));
  L.cnt = o;  o = align256(o + sizeof(int) * nseg);
  L.off = o;  o = align256(o + sizeof(int) * (nseg + 1));
  L.pos = o;  o = align256(o + sizeof(int) * size_t(T) * K);
  L.perm = o; o = align256(o + sizeof(int) * size_t(L.mcap));
  L.done = o; o = align256(o + sizeof(int) * (nseg + kClaimSlots));
  L.pscr = o; o = align256(o + (T * K > kPermSingleMax ? sizeof(int) * kPermScrInts : 0));
  L.xp = o;   o = align256(o + (L.tc ? size_t(L.mcap) * d * 2 : 0));
  L.h = o;    o = align256(o + size_t(L.mcap) * w * (dtype == MCFT_BF16 ? 2 : 4));
  L.o = o;    o = align256(o + size_t(L.ks) * L.mcap * d * 4);
  L.u13 = o;  o = align256(o + size_t(L.mcap) * 2 * lrank * 4);
  L.u2 = o;   o = align256(o + size_t(L.mcap) * lrank * 4);
  L.total = o;
  return L;
}

}  // namespace mcft

using namespace mcft;

// ------------------------------------------------------------------------------------------------
// Expert cache object

struct mcft_cache {
  int L = 0, E = 0, B = 0, max_assign = 0, n_staging = 0, device = 0, policy = 0;
  size_t expert_bytes = 0;
  std::vector<const void*> host_experts;  // [L*E] pinned host blocks (empty: accounting only)
  int32_t* d_tag = nullptr;
  int64_t* d_last = nullptr;
  int64_t* d_ins = nullptr;
  int64_t* d_freq = nullptr;
  int64_t* d_step = nullptr;
  unsigned long long* d_cnt = nullptr;
  int32_t* h_miss = nullptr;  // host-mapped [L][miss_stride]
  int32_t* d_miss = nullptr;  // device alias of h_miss
  int miss_stride = 0;
  int32_t* d_miss_dev = nullptr;            // device-memory copy [L][miss_stride]
  unsigned long long* d_ptr_tab = nullptr;  // [L*E] block address of each selected expert
  unsigned long long* d_ready = nullptr;    // [L] hit mask of the last step
  unsigned long long* d_stream = nullptr;   // [L] miss mask of the last step
  unsigned* d_landed = nullptr;  // [L][E][ppe] epoch stamps of the demand fetch's landed pieces
  unsigned* d_fctr = nullptr;    // [L][2] role and piece counters of that fetching FFN launch
  int ppe = 0;                   // fetch pieces per expert block
  unsigned long long* d_host_src = nullptr; // [L*E] device-visible addresses of the host blocks
  unsigned long long* d_pfmask = nullptr;   // [L] experts loaded by a prefetch since the last step
  unsigned long long* d_pf_cancel = nullptr;  // [L] prefetched experts the next step dropped
  unsigned long long* d_pf_moved = nullptr;   // [L] bytes the prefetch fetches copied
  int32_t* d_pf_list = nullptr;             // [L][1 + E] fetch list of the last prefetch
  unsigned long long* d_pf_tab = nullptr;   // [L*E] destinations of the last prefetch's loads
  char* d_slots = nullptr;    // [L*B] expert blocks
  char* d_staging = nullptr;  // [n_staging] expert blocks
  std::vector<cudaEvent_t> ev_step;  // per layer: recorded after its cache step
  std::vector<cudaEvent_t> ev_pf_step, ev_pf_done;  // per layer: after a prefetch decision / fetch
  // per layer: 0 no prefetch outstanding, 1 decided (fetch not yet enqueued), 2 fetch enqueued and
  // not yet waited for by a compute stream
  std::vector<int> pf_state;
  cudaEvent_t ev_copy = nullptr;
  bool device_fetch = false;  // every host block has a device-visible address
};

namespace {

void cache_free(mcft_cache* c) {
  if (!c) return;
  cudaFree(c->d_tag);
  cudaFree(c->d_last);
  cudaFree(c->d_ins);
  cudaFree(c->d_freq);
  cudaFree(c->d_step);
  cudaFree(c->d_cnt);
  if (c->h_miss) cudaFreeHost(c->h_miss);
  cudaFree(c->d_slots);
  cudaFree(c->d_staging);
  cudaFree(c->d_miss_dev);
  cudaFree(c->d_ptr_tab);
  cudaFree(c->d_ready);
  cudaFree(c->d_stream);
  cudaFree(c->d_landed);
  cudaFree(c->d_fctr);
  cudaFree(c->d_host_src);
  cudaFree(c->d_pfmask);
  cudaFree(c->d_pf_cancel);
  cudaFree(c->d_pf_moved);
  cudaFree(c->d_pf_list);
  cudaFree(c->d_pf_tab);
  for (const auto* v : {&c->ev_step, &c->ev_pf_step, &c->ev_pf_done})
    for (cudaEvent_t e : *v)
      if (e) cudaEventDestroy(e);
  if (c->ev_copy) cudaEventDestroy(c->ev_copy);
  delete c;
}

const char* loc_ptr(const mcft_cache* c, int layer, int loc) {
  if (loc < 0 || !c->d_slots) return nullptr;
  if (loc < c->B) return c->d_slots + (size_t(layer) * c->B + loc) * c->expert_bytes;
  return c->d_staging + size_t(loc - c->B) * c->expert_bytes;
}

struct CacheStateHeader {
  uint32_t magic, L, E, B, policy, pad;
};
constexpr uint32_t kStateMagic = 0x4d434656u;

// Bytes of the exported state: header, tag [L*B] i32, last and ins [L*B] i64, freq [L*E] i64,
// step [L] i64, counters [L*5] u64, prefetch mask [L] u64.
size_t state_bytes(const mcft_cache* c) {
  const size_t LB = size_t(c->L) * c->B, LE = size_t(c->L) * c->E;
  return sizeof(CacheStateHeader) + LB * 4 + LB * 8 * 2 + LE * 8 + size_t(c->L) * 8 +
         size_t(c->L) * 8 * kCacheCounters + size_t(c->L) * 8;
}

// Enqueue on `copy` the fetch of every prefetch decided but not yet fetched (in layer order).
mcft_status enqueue_prefetch_fetches(mcft_cache* c, cudaStream_t copy) {
  for (int l = 0; l < c->L; ++l) {
    if (c->pf_state[l] != 1) continue;
    MCFT_CUDA(cudaStreamWaitEvent(copy, c->ev_pf_step[l], 0));
    FetchArgs fe{c->d_pf_list + size_t(l) * (1 + c->E), c->d_host_src + size_t(l) * c->E,
                 c->d_pf_tab + size_t(l) * c->E, c->expert_bytes, c->d_pf_cancel + l,
                 c->d_pf_moved + l};
    cudaError_t e = launch_fetch(fe, fetch_blocks(), copy, true);
    if (e != cudaSuccess) return cuda_fail(e, "prefetch fetch kernel launch");
    MCFT_CUDA(cudaEventRecord(c->ev_pf_done[l], copy));
    c->pf_state[l] = 2;
  }
  return MCFT_OK;
}

}  // namespace

extern "C" {

int mcft_version(void) { return 200; }

mcft_status mcft_test_inject(int fail_pinned_allocs, int fail_expert_copies,
                             unsigned long long wait_limit_ns, int withhold_gemm13) {
  if (fail_pinned_allocs < 0 || fail_expert_copies < 0)
    return fail(MCFT_ERR_INVALID, "failure counts must be >= 0");
  g_inject_pinned.store(fail_pinned_allocs);
  g_inject_copy.store(fail_expert_copies);
  g_inject_wait_ns.store(wait_limit_ns);
  g_inject_withhold.store(withhold_gemm13 ? 1 : 0);
  return MCFT_OK;
}

mcft_status mcft_set_tc_tiles(int mode) {
  if (mode != MCFT_TC_TILES_ONE_CTA && mode != MCFT_TC_TILES_CTA_PAIR)
    return fail(MCFT_ERR_INVALID, "tile mode %d is neither one-CTA (0) nor CTA-pair (1)", mode);
  g_tc_tiles.store(mode);
  return MCFT_OK;
}

const char* mcft_last_error(void) { return g_last_error.c_str(); }

mcft_status mcft_device_error(mcft_stream_t stream) {
  unsigned* p = device_error_word();
  if (!p) return fail(MCFT_ERR_CUDA, "cannot locate the device error word");
  unsigned v = 0;
  MCFT_CUDA(cudaStreamSynchronize(stream));
  MCFT_CUDA(cudaMemcpyAsync(&v, p, sizeof(v), cudaMemcpyDeviceToHost, stream));
  MCFT_CUDA(cudaMemsetAsync(p, 0, sizeof(unsigned), stream));
  MCFT_CUDA(cudaStreamSynchronize(stream));
  if (v == 0) return MCFT_OK;
  return fail(static_cast<mcft_status>(v), "device error %u reported by a kernel", v);
}

mcft_status mcft_route(const mcft_layer_desc* desc, const void* x, int T, const void* w_router,
                       int mode, const uint8_t* mask, const float* prior, int32_t* idx, float* gate,
                       mcft_stream_t stream) {
  mcft::NvtxRange nvtx_range("mcft_route");
  mcft_status st = check_desc(desc);
  if (st != MCFT_OK) return st;
  if (T < 0) return fail(MCFT_ERR_INVALID, "T = %d < 0", T);
  if (mode != MCFT_ROUTE_TOPK && mode != MCFT_ROUTE_HARD_MASK && mode != MCFT_ROUTE_SOFT_PRIOR)
    return fail(MCFT_ERR_INVALID, "unknown routing mode %d", mode);
  RouteArgs a{};
  if (mode == MCFT_ROUTE_HARD_MASK) {
    if (!mask) return fail(MCFT_ERR_INVALID, "hard-mask routing needs a mask");
    int ones = 0;
    for (int e = 0; e < desc->E; ++e) {
      if (mask[e] > 1) return fail(MCFT_ERR_INVALID, "mask[%d] = %d is not 0 or 1", e, mask[e]);
      ones += mask[e];
      a.mask[e] = mask[e];
    }
    if (ones < desc->K)
      return fail(MCFT_ERR_INVALID, "mask keeps %d experts, fewer than K = %d", ones, desc->K);
  } else if (mode == MCFT_ROUTE_SOFT_PRIOR) {
    if (!prior) return fail(MCFT_ERR_INVALID, "soft-prior routing needs a prior");
    for (int e = 0; e < desc->E; ++e) {
      const float v = prior[e];
      if (!(v > 0.f) || v > 3.4e38f)
        return fail(MCFT_ERR_INVALID, "prior[%d] = %g must be positive and finite", e, double(v));
      a.prior[e] = v;
    }
  }
  if (T == 0) return MCFT_OK;
  if (!x || !w_router || !idx || !gate) return fail(MCFT_ERR_INVALID, "NULL tensor pointer");
  if ((reinterpret_cast<uintptr_t>(x) | reinterpret_cast<uintptr_t>(w_router)) & 15u)
    return fail(MCFT_ERR_INVALID, "x and w_router must be 16-byte aligned");
  a.x = x;
  a.w_router = w_router;
  a.T = T;
  a.d = desc->d;
  a.E = desc->E;
  a.K = desc->K;
  a.mode = mode;
  a.gate_mode = desc->gate;
  a.idx = idx;
  a.gate = gate;
  a.err = device_error_word();
  cudaError_t e = launch_route(a, desc->dtype, stream);
  if (e != cudaSuccess) return cuda_fail(e, "route kernel launch");
  return MCFT_OK;
}

}  // extern "C"

namespace {

size_t workspace_bytes(const mcft_layer_desc* desc, int T_max, int lrank) {
  // the largest layout over every T <= T_max (the decode path's split depends on T)
  size_t best = 0;
  const int upto = T_max < 64 ? T_max : 64;
  for (int T = 0; T <= upto + 1; ++T) {
    const int t = T <= upto ? T : T_max;
    const WsLayout L =
        ws_layout(desc->d, desc->E, desc->K, desc->w, desc->n_shared, desc->dtype, t, lrank);
    if (L.total > best) best = L.total;
  }
  return best;
}

mcft_status check_lora(int rank, float scale) {
  if (rank != 8 && rank != 16)
    return fail(MCFT_ERR_UNSUPPORTED, "LoRA rank %d (supported: 8, 16)", rank);
  if (!(scale == scale) || scale > 3.4e38f || scale < -3.4e38f)
    return fail(MCFT_ERR_INVALID, "LoRA scale must be finite");
  return MCFT_OK;
}

struct LoraArgs {
  const void* const* expert;  // host [E] adapter blocks (NULL entries: no adapter)
  const void* const* shared;  // host [S]
  int rank;
  float scale;
};

// Permutation, grouped SwiGLU FFN (optionally with LoRA adapters) and combine.
mcft_status forward_impl(const mcft_layer_desc* desc, const void* x, int T, const int32_t* idx,
                         const float* gate, const void* const* experts, const void* const* shared,
                         const LoraArgs* lora, void* y, void* workspace, size_t ws_bytes,
                         cudaStream_t stream) {
  mcft_status st = check_desc(desc);
  if (st != MCFT_OK) return st;
  if (T < 0) return fail(MCFT_ERR_INVALID, "T = %d < 0", T);
  if (T == 0) return MCFT_OK;
  if (!x || !idx || !gate || !experts || !y || !workspace)
    return fail(MCFT_ERR_INVALID, "NULL pointer argument");
  if (desc->n_shared > 0 && !shared) return fail(MCFT_ERR_INVALID, "shared is NULL");
  if (reinterpret_cast<uintptr_t>(workspace) & 255u)
    return fail(MCFT_ERR_INVALID, "workspace must be 256-byte aligned");
  if ((reinterpret_cast<uintptr_t>(x) | reinterpret_cast<uintptr_t>(y)) & 15u)
    return fail(MCFT_ERR_INVALID, "x and y must be 16-byte aligned");
  const int E = desc->E, S = desc->n_shared, K = desc->K;
  const int lrank = lora ? lora->rank : 0;
  const WsLayout L = ws_layout(desc->d, E, K, desc->w, S, desc->dtype, T, lrank);
  if (ws_bytes < L.total)
    return fail(MCFT_ERR_INVALID, "workspace of %zu bytes < %zu needed", ws_bytes, L.total);
  for (int e = 0; e < E; ++e)
    if (reinterpret_cast<uintptr_t>(experts[e]) & 15u)
      return fail(MCFT_ERR_INVALID, "expert %d block is not 16-byte aligned", e);
  for (int s = 0; s < S; ++s)
    if (!shared[s] || (reinterpret_cast<uintptr_t>(shared[s]) & 15u))
      return fail(MCFT_ERR_INVALID, "shared expert %d block is NULL or misaligned", s);
  if (lora) {
    if (!lora->expert || (S > 0 && !lora->shared))
      return fail(MCFT_ERR_INVALID, "NULL adapter array");
    for (int i = 0; i < E + S; ++i) {
      const void* p = i < E ? lora->expert[i] : lora->shared[i - E];
      if (reinterpret_cast<uintptr_t>(p) & 15u)
        return fail(MCFT_ERR_INVALID, "adapter block %d is not 16-byte aligned", i);
    }
  }

  char* ws = static_cast<char*>(workspace);
  WsHeader* hdr = reinterpret_cast<WsHeader*>(ws + L.hdr);
  int* cnt = reinterpret_cast<int*>(ws + L.cnt);
  int* off = reinterpret_cast<int*>(ws + L.off);
  int* pos = reinterpret_cast<int*>(ws + L.pos);
  int* perm = reinterpret_cast<int*>(ws + L.perm);
  unsigned* err = device_error_word();

  int* done = reinterpret_cast<int*>(ws + L.done);
  PermuteArgs pa{idx, T, K, E, S, L.pad, L.mcap, hdr, cnt, off, pos, perm, err, done,
                 T * K > kPermSingleMax ? reinterpret_cast<int*>(ws + L.pscr) : nullptr};
  cudaError_t e = launch_permute(pa, stream);
  if (e != cudaSuccess) return cuda_fail(e, "permute kernel launch");

  FfnArgs fa{};
  fa.x = x;
  fa.off = off;
  fa.perm = perm;
  fa.hdr = hdr;
  fa.done = done;
  for (int i = 0; i < E; ++i) fa.wblk[i] = experts[i];
  for (int s = 0; s < S; ++s) fa.wblk[E + s] = shared[s];
  fa.h = ws + L.h;
  fa.o = reinterpret_cast<float*>(ws + L.o);
  fa.o_plane = size_t(L.mcap) * desc->d;
  fa.ksplit = L.ks;
  fa.T = T;
  fa.d = desc->d;
  fa.w = desc->w;
  fa.nseg = E + S;
  fa.E = E;
  fa.err = err;
  LoraDownArgs la{};
  if (lora) {
    for (int i = 0; i < E; ++i) fa.lblk[i] = lora->expert[i];
    for (int s = 0; s < S; ++s) fa.lblk[E + s] = lora->shared[s];
    fa.lrank = lrank;
    fa.lscale = lora->scale;
    fa.u13 = reinterpret_cast<float*>(ws + L.u13);
    fa.u2 = reinterpret_cast<float*>(ws + L.u2);
    const LoraOffsets lo = lora_offsets(desc->d, desc->w, lrank);
    la.row_tok = perm;
    la.off = off;
    la.hdr = hdr;
    la.nseg = E + S;
    for (int i = 0; i < E + S; ++i) la.lblk[i] = fa.lblk[i];
    la.r = lrank;
    // u13[q] = [A1 x ; A3 x] for the token of every permuted row
    la.in = x;
    la.in_stride = size_t(desc->d);
    la.by_token = 1;
    la.a_off0 = lo.a1;
    la.a_off1 = lo.a3;
    la.K = desc->d;
    la.u = const_cast<float*>(fa.u13);
    la.ustride = 2 * lrank;
    if (!L.tc) {  // the tcgen05 path projects the gathered rows instead, after the gather
      e = launch_lora_down(la, desc->dtype, 2 * lrank, L.mcap, stream);
      if (e != cudaSuccess) return cuda_fail(e, "LoRA kernel launch");
    }
  }
  auto ffn = [&](int stages) -> cudaError_t {
    if (L.tc) return launch_ffn_tc(fa, ws + L.xp, L.mcap, L.pad, num_sms(), stream, stages);
    if (L.decode) return launch_ffn_decode(fa, num_sms(), stream, stages);
    return launch_ffn_rowwise(fa, desc->dtype, num_sms(), stream, stages);
  };
  if (L.tc) {
    GatherArgs ga{x, perm, hdr, ws + L.xp, desc->d, L.mcap};
    e = launch_gather(ga, stream);
    if (e != cudaSuccess) return cuda_fail(e, "gather kernel launch");
    if (lora) {  // U13, GEMM13, U2 (from h), GEMM2
      e = launch_lora_down_tc(fa, ws + L.xp, L.mcap, num_sms(), stream, 1);
      if (e == cudaSuccess) e = ffn(1);
      if (e == cudaSuccess) e = launch_lora_down_tc(fa, ws + L.xp, L.mcap, num_sms(), stream, 2);
      if (e == cudaSuccess) e = ffn(2);
      if (e != cudaSuccess) return cuda_fail(e, "LoRA expert GEMM launch");
    }
  }
  if (!(lora && L.tc)) {
    e = ffn(lora ? 1 : 3);
    if (e != cudaSuccess) return cuda_fail(e, "expert FFN launch");
  }
  if (lora && !L.tc) {
    // u2[q] = A2 h_q for every permuted row, then the down projection with its adapter
    const LoraOffsets lo = lora_offsets(desc->d, desc->w, lrank);
    la.in = fa.h;
    la.in_stride = size_t(desc->w);
    la.by_token = 0;
    la.a_off0 = lo.a2;
    la.a_off1 = 0;
    la.K = desc->w;
    la.u = const_cast<float*>(fa.u2);
    la.ustride = lrank;
    e = launch_lora_down(la, desc->dtype, lrank, L.mcap, stream);
    if (e != cudaSuccess) return cuda_fail(e, "LoRA kernel launch");
    e = ffn(2);
    if (e != cudaSuccess) return cuda_fail(e, "expert FFN launch");
  }
  CombineArgs ca{fa.o, gate, pos, off, hdr, y, T, desc->d, K, E, S, L.ks, fa.o_plane};
  e = launch_combine(ca, desc->dtype, stream);
  if (e != cudaSuccess) return cuda_fail(e, "combine kernel launch");
  return MCFT_OK;
}

}  // namespace

extern "C" {

mcft_status mcft_moe_workspace_size(const mcft_layer_desc* desc, int T_max, size_t* bytes) {
  mcft_status st = check_desc(desc);
  if (st != MCFT_OK) return st;
  if (T_max < 0 || !bytes) return fail(MCFT_ERR_INVALID, "T_max < 0 or bytes is NULL");
  *bytes = workspace_bytes(desc, T_max, 0);
  return MCFT_OK;
}

mcft_status mcft_moe_workspace_size_lora(const mcft_layer_desc* desc, int lora_rank, int T_max,
                                         size_t* bytes) {
  mcft_status st = check_desc(desc);
  if (st != MCFT_OK) return st;
  st = check_lora(lora_rank, 1.f);
  if (st != MCFT_OK) return st;
  if (T_max < 0 || !bytes) return fail(MCFT_ERR_INVALID, "T_max < 0 or bytes is NULL");
  *bytes = workspace_bytes(desc, T_max, lora_rank);
  return MCFT_OK;
}

mcft_status mcft_moe_forward(const mcft_layer_desc* desc, const void* x, int T, const int32_t* idx,
                             const float* gate, const void* const* experts,
                             const void* const* shared, void* y, void* workspace, size_t ws_bytes,
                             mcft_stream_t stream) {
  mcft::NvtxRange nvtx_range("mcft_moe_forward");
  return forward_impl(desc, x, T, idx, gate, experts, shared, nullptr, y, workspace, ws_bytes,
                      stream);
}

mcft_status mcft_moe_forward_lora(const mcft_layer_desc* desc, const void* x, int T,
                                  const int32_t* idx, const float* gate,
                                  const void* const* experts, const void* const* shared,
                                  const void* const* expert_lora, const void* const* shared_lora,
                                  int lora_rank, float lora_scale, void* y, void* workspace,
                                  size_t ws_bytes, mcft_stream_t stream) {
  mcft::NvtxRange nvtx_range("mcft_moe_forward_lora");
  mcft_status st = check_lora(lora_rank, lora_scale);
  if (st != MCFT_OK) return st;
  const LoraArgs la{expert_lora, shared_lora, lora_rank, lora_scale};
  return forward_impl(desc, x, T, idx, gate, experts, shared, &la, y, workspace, ws_bytes, stream);
}

// ------------------------------------------------------------------------------------------------

mcft_status mcft_cache_create(int L, int E, int B, size_t expert_bytes,
                              const void* const* host_experts, int max_assign, int policy,
                              mcft_cache** out) {
  if (!out) return fail(MCFT_ERR_INVALID, "out is NULL");
  *out = nullptr;
  if (L <= 0) return fail(MCFT_ERR_INVALID, "L = %d must be positive", L);
  if (E <= 1) return fail(MCFT_ERR_INVALID, "E = %d must be at least 2", E);
  if (E > kMaxE) return fail(MCFT_ERR_UNSUPPORTED, "E = %d > %d", E, kMaxE);
  if (B < 1 || B >= E) return fail(MCFT_ERR_INVALID, "need 1 <= B < E (B = %d, E = %d)", B, E);
  if (max_assign < 1) return fail(MCFT_ERR_INVALID, "max_assign = %d must be positive", max_assign);
  if (policy != MCFT_CACHE_LRU && policy != MCFT_CACHE_LFU && policy != MCFT_CACHE_FIFO)
    return fail(MCFT_ERR_INVALID, "unknown cache policy %d", policy);
  if (host_experts) {
    if (expert_bytes == 0 || expert_bytes % 16)
      return fail(MCFT_ERR_INVALID, "expert_bytes = %zu must be a positive multiple of 16", expert_bytes);
    for (int i = 0; i < L * E; ++i)
      if (!host_experts[i]) return fail(MCFT_ERR_INVALID, "host expert %d is NULL", i);
  }
  mcft_cache* c = new mcft_cache();
  c->L = L;
  c->E = E;
  c->B = B;
  c->max_assign = max_assign;
  c->policy = policy;
  c->expert_bytes = expert_bytes;
  c->device = current_device();
  c->miss_stride = (1 + 3 * E + 3) & ~3;
  const int stg = E - B < max_assign ? E - B : max_assign;
#define MCFT_CACHE_CUDA(call)                    \
  do {                                           \
    cudaError_t e_ = (call);                     \
    if (e_ != cudaSuccess) {                     \
      cache_free(c);                             \
      return cuda_fail(e_, #call);               \
    }                                            \
  } while (0)
  MCFT_CACHE_CUDA(cudaMalloc(&c->d_tag, sizeof(int32_t) * L * B));
  MCFT_CACHE_CUDA(cudaMalloc(&c->d_last, sizeof(int64_t) * L * B));
  MCFT_CACHE_CUDA(cudaMalloc(&c->d_ins, sizeof(int64_t) * L * B));
  MCFT_CACHE_CUDA(cudaMalloc(&c->d_freq, sizeof(int64_t) * L * E));
  MCFT_CACHE_CUDA(cudaMalloc(&c->d_step, sizeof(int64_t) * L));
  MCFT_CACHE_CUDA(cudaMalloc(&c->d_cnt, sizeof(unsigned long long) * L * kCacheCounters));
  MCFT_CACHE_CUDA(cudaMalloc(&c->d_pfmask, sizeof(unsigned long long) * L));
  MCFT_CACHE_CUDA(cudaMemset(c->d_pfmask, 0, sizeof(unsigned long long) * L));
  MCFT_CACHE_CUDA(cudaMalloc(&c->d_pf_cancel, sizeof(unsigned long long) * L));
  MCFT_CACHE_CUDA(cudaMemset(c->d_pf_cancel, 0, sizeof(unsigned long long) * L));
  MCFT_CACHE_CUDA(cudaMalloc(&c->d_pf_moved, sizeof(unsigned long long) * L));
  MCFT_CACHE_CUDA(cudaMemset(c->d_pf_moved, 0, sizeof(unsigned long long) * L));
  MCFT_CACHE_CUDA(cudaMalloc(&c->d_pf_list, sizeof(int32_t) * L * (1 + E)));
  MCFT_CACHE_CUDA(cudaMemset(c->d_pf_list, 0, sizeof(int32_t) * L * (1 + E)));
  MCFT_CACHE_CUDA(cudaMalloc(&c->d_pf_tab, sizeof(unsigned long long) * L * E));
  MCFT_CACHE_CUDA(cudaMemset(c->d_pf_tab, 0, sizeof(unsigned long long) * L * E));
  MCFT_CACHE_CUDA(cudaMemset(c->d_tag, 0xff, sizeof(int32_t) * L * B));  // -1 = empty
  MCFT_CACHE_CUDA(cudaMemset(c->d_last, 0xff, sizeof(int64_t) * L * B));
  MCFT_CACHE_CUDA(cudaMemset(c->d_ins, 0xff, sizeof(int64_t) * L * B));
  MCFT_CACHE_CUDA(cudaMemset(c->d_freq, 0, sizeof(int64_t) * L * E));
  MCFT_CACHE_CUDA(cudaMemset(c->d_step, 0, sizeof(int64_t) * L));
  MCFT_CACHE_CUDA(cudaMemset(c->d_cnt, 0, sizeof(unsigned long long) * L * kCacheCounters));
  MCFT_CACHE_CUDA(host_alloc_mapped(reinterpret_cast<void**>(&c->h_miss),
                                    sizeof(int32_t) * L * c->miss_stride));
  memset(c->h_miss, 0, sizeof(int32_t) * L * c->miss_stride);
  MCFT_CACHE_CUDA(cudaHostGetDevicePointer(reinterpret_cast<void**>(&c->d_miss), c->h_miss, 0));
  MCFT_CACHE_CUDA(cudaMalloc(&c->d_miss_dev, sizeof(int32_t) * L * c->miss_stride));
  MCFT_CACHE_CUDA(cudaMemset(c->d_miss_dev, 0, sizeof(int32_t) * L * c->miss_stride));
  MCFT_CACHE_CUDA(cudaMalloc(&c->d_ptr_tab, sizeof(unsigned long long) * L * E));
  MCFT_CACHE_CUDA(cudaMemset(c->d_ptr_tab, 0, sizeof(unsigned long long) * L * E));
  MCFT_CACHE_CUDA(cudaMalloc(&c->d_ready, sizeof(unsigned long long) * L));
  MCFT_CACHE_CUDA(cudaMemset(c->d_ready, 0, sizeof(unsigned long long) * L));
  MCFT_CACHE_CUDA(cudaMalloc(&c->d_stream, sizeof(unsigned long long) * L));
  MCFT_CACHE_CUDA(cudaMemset(c->d_stream, 0, sizeof(unsigned long long) * L));
  if (host_experts) {
    c->host_experts.assign(host_experts, host_experts + size_t(L) * E);
    c->n_staging = stg;
    MCFT_CACHE_CUDA(cudaMalloc(&c->d_slots, expert_bytes * size_t(L) * B));
    // stamps start below every epoch (steps count from 1)
    c->ppe = int((expert_bytes + kFetchPiece - 1) / kFetchPiece);
    MCFT_CACHE_CUDA(cudaMalloc(&c->d_landed, sizeof(unsigned) * size_t(L) * E * c->ppe));
    MCFT_CACHE_CUDA(cudaMemset(c->d_landed, 0, sizeof(unsigned) * size_t(L) * E * c->ppe));
    MCFT_CACHE_CUDA(cudaMalloc(&c->d_fctr, sizeof(unsigned) * 2 * size_t(L)));
    MCFT_CACHE_CUDA(cudaMemset(c->d_fctr, 0, sizeof(unsigned) * 2 * size_t(L)));
    if (stg > 0) MCFT_CACHE_CUDA(cudaMalloc(&c->d_staging, expert_bytes * size_t(stg)));
    // device-visible addresses of the pinned host blocks, for the device-driven fetch
    std::vector<unsigned long long> src(size_t(L) * E);
    for (size_t i = 0; i < src.size(); ++i) {
      void* dp = nullptr;
      if (cudaHostGetDevicePointer(&dp, const_cast<void*>(host_experts[i]), 0) != cudaSuccess) {
        cudaGetLastError();
        dp = nullptr;  // not mapped: only the copy-engine fetch can serve this cache
      }
      src[i] = reinterpret_cast<unsigned long long>(dp);
    }
    MCFT_CACHE_CUDA(cudaMalloc(&c->d_host_src, sizeof(unsigned long long) * L * E));
    MCFT_CACHE_CUDA(cudaMemcpy(c->d_host_src, src.data(), sizeof(unsigned long long) * L * E,
                               cudaMemcpyHostToDevice));
    c->device_fetch = true;
    for (auto v : src) c->device_fetch = c->device_fetch && v != 0;
  }
  c->ev_step.assign(L, nullptr);
  c->ev_pf_step.assign(L, nullptr);
  c->ev_pf_done.assign(L, nullptr);
  c->pf_state.assign(L, 0);
  for (int l = 0; l < L; ++l) {
    MCFT_CACHE_CUDA(cudaEventCreateWithFlags(&c->ev_step[l], cudaEventDisableTiming));
    MCFT_CACHE_CUDA(cudaEventCreateWithFlags(&c->ev_pf_step[l], cudaEventDisableTiming));
    MCFT_CACHE_CUDA(cudaEventCreateWithFlags(&c->ev_pf_done[l], cudaEventDisableTiming));
  }
  MCFT_CACHE_CUDA(cudaEventCreateWithFlags(&c->ev_copy, cudaEventDisableTiming));
  MCFT_CACHE_CUDA(cudaDeviceSynchronize());
#undef MCFT_CACHE_CUDA
  *out = c;
  return MCFT_OK;
}

mcft_status mcft_cache_step(mcft_cache* c, int layer, const int32_t* idx, int T, int K,
                            mcft_stream_t stream) {
  mcft::NvtxRange nvtx_range("mcft_cache_step");
  if (!c || !idx) return fail(MCFT_ERR_INVALID, "NULL cache or idx");
  if (layer < 0 || layer >= c->L) return fail(MCFT_ERR_INVALID, "layer %d out of range", layer);
  if (T < 1 || K < 1 || K > c->E) return fail(MCFT_ERR_INVALID, "bad T = %d or K = %d", T, K);
  if (T * K > c->max_assign)
    return fail(MCFT_ERR_INVALID, "T*K = %d exceeds max_assign = %d", T * K, c->max_assign);
  CacheStepArgs a{idx, T * K, c->E, c->B, layer, c->policy, c->d_tag, c->d_last, c->d_ins,
                  c->d_freq, c->d_step, c->d_cnt, c->d_pfmask, c->d_pf_cancel,
                  c->d_miss + size_t(layer) * c->miss_stride,
                  c->d_miss_dev + size_t(layer) * c->miss_stride,
                  c->d_ptr_tab + size_t(layer) * c->E, c->d_ready + layer, c->d_stream + layer,
                  c->d_fctr ? c->d_fctr + 2 * size_t(layer) : nullptr,
                  c->d_slots ? c->d_slots + size_t(layer) * c->B * c->expert_bytes : nullptr,
                  c->d_staging, c->expert_bytes, device_error_word()};
  cudaError_t e = launch_cache_step(a, stream);
  if (e != cudaSuccess) return cuda_fail(e, "cache step launch");
  MCFT_CUDA(cudaEventRecord(c->ev_step[layer], stream));
  return MCFT_OK;
}

mcft_status mcft_read_probe(const void* buf, size_t bytes, int pattern, int row_bytes, int blocks,
                            unsigned* sink, mcft_stream_t stream) {
  if (!buf || !sink) return fail(MCFT_ERR_INVALID, "NULL pointer");
  if (reinterpret_cast<uintptr_t>(buf) % 16) return fail(MCFT_ERR_INVALID, "buf must be 16-byte aligned");
  if (pattern != 0 && pattern != 1) return fail(MCFT_ERR_INVALID, "pattern %d is not 0 or 1", pattern);
  if (blocks < 1 || blocks > 65535) return fail(MCFT_ERR_INVALID, "blocks = %d out of range", blocks);
  if (pattern == 0 && bytes % 16) return fail(MCFT_ERR_INVALID, "bytes = %zu is not a multiple of 16", bytes);
  if (pattern == 1 && (row_bytes <= 0 || row_bytes % 128 || bytes % (size_t(32) * row_bytes)))
    return fail(MCFT_ERR_INVALID, "pattern 1 needs row_bytes a positive multiple of 128 and bytes "
                "a multiple of 32 rows");
  if (bytes == 0) return MCFT_OK;
  const cudaError_t e = launch_read_probe(buf, bytes, pattern, row_bytes, blocks, sink, stream);
  if (e != cudaSuccess) return cuda_fail(e, "read probe launch");
  return MCFT_OK;
}

mcft_status mcft_host_copy(void* dst, const void* host_src, size_t bytes, int blocks,
                           mcft_stream_t stream) {
  if (!dst || !host_src) return fail(MCFT_ERR_INVALID, "NULL pointer");
  if ((reinterpret_cast<uintptr_t>(dst) | reinterpret_cast<uintptr_t>(host_src)) % 16)
    return fail(MCFT_ERR_INVALID, "pointers must be 16-byte aligned");
  if (bytes % 16) return fail(MCFT_ERR_INVALID, "bytes = %zu is not a multiple of 16", bytes);
  if (blocks < 1 || blocks > 65535) return fail(MCFT_ERR_INVALID, "blocks = %d out of range", blocks);
  if (bytes == 0) return MCFT_OK;
  void* src = nullptr;
  if (cudaHostGetDevicePointer(&src, const_cast<void*>(host_src), 0) != cudaSuccess) {
    cudaGetLastError();
    return fail(MCFT_ERR_INVALID, "host_src is not host memory the device can address");
  }
  const cudaError_t e = launch_host_copy(dst, src, bytes, blocks, stream);
  if (e != cudaSuccess) return cuda_fail(e, "host copy kernel launch");
  return MCFT_OK;
}

mcft_status mcft_fetch_experts(mcft_cache* c, int layer, mcft_stream_t compute_stream,
                               mcft_stream_t copy_stream, const void** expert_ptrs) {
  mcft::NvtxRange nvtx_range("mcft_fetch_experts");
  if (!c || !expert_ptrs) return fail(MCFT_ERR_INVALID, "NULL cache or expert_ptrs");
  if (layer < 0 || layer >= c->L) return fail(MCFT_ERR_INVALID, "layer %d out of range", layer);
  // The miss list is known only once routing and the cache decision have run.
  MCFT_CUDA(cudaEventSynchronize(c->ev_step[layer]));
  const int32_t* m = c->h_miss + size_t(layer) * c->miss_stride;
  const int E = c->E;
  const int nm = m[0];
  const int32_t* m_exp = m + 1;
  const int32_t* loc_of = m + 1 + 2 * E;
  for (int e = 0; e < E; ++e) expert_ptrs[e] = loc_ptr(c, layer, loc_of[e]);
  // a prefetch of this layer decided before the step lands before the step's own copies
  if (c->pf_state[layer] == 1) {
    mcft_status st = enqueue_prefetch_fetches(c, copy_stream);
    if (st != MCFT_OK) return st;
  }
  if (c->pf_state[layer] == 2) {
    MCFT_CUDA(cudaStreamWaitEvent(compute_stream, c->ev_pf_done[layer], 0));
    c->pf_state[layer] = 0;
  }
  if (c->d_slots && nm > 0) {
    // Every earlier use of these slots finished before the cache step's event (same stream).
    for (int i = 0; i < nm; ++i) {
      const int e = m_exp[i];
      if (e < 0 || e >= E) return fail(MCFT_ERR_INVALID, "corrupt miss list");
      const char* dst = loc_ptr(c, layer, loc_of[e]);
      MCFT_CUDA(expert_copy(const_cast<char*>(dst), c->host_experts[size_t(layer) * E + e],
                            c->expert_bytes, copy_stream));
    }
    MCFT_CUDA(cudaEventRecord(c->ev_copy, copy_stream));
    MCFT_CUDA(cudaStreamWaitEvent(compute_stream, c->ev_copy, 0));
  }
  // prefetches of later layers stream in behind this layer's copies
  return enqueue_prefetch_fetches(c, copy_stream);
}

mcft_status mcft_cache_prefetch(mcft_cache* c, int layer, const int32_t* idx_pred, int T, int K,
                                int n_max, mcft_stream_t stream) {
  mcft::NvtxRange nvtx_range("mcft_cache_prefetch");
  if (!c || !idx_pred) return fail(MCFT_ERR_INVALID, "NULL cache or idx_pred");
  if (layer < 0 || layer >= c->L) return fail(MCFT_ERR_INVALID, "layer %d out of range", layer);
  if (T < 1 || K < 1 || K > c->E) return fail(MCFT_ERR_INVALID, "bad T = %d or K = %d", T, K);
  if (T * K > c->max_assign)
    return fail(MCFT_ERR_INVALID, "T*K = %d exceeds max_assign = %d", T * K, c->max_assign);
  if (n_max < 1 || n_max > c->B)
    return fail(MCFT_ERR_INVALID, "n_max = %d must be in [1, B = %d]", n_max, c->B);
  if (c->d_slots && !c->device_fetch)
    return fail(MCFT_ERR_UNSUPPORTED, "prefetch needs host blocks with device-visible addresses");
  if (c->pf_state[layer] == 1)
    return fail(MCFT_ERR_INVALID, "the previous prefetch of layer %d was never fetched (run a "
                "forward or mcft_fetch_experts first)", layer);
  // the previous prefetch's list is rewritten and its slots may be chosen again
  if (c->pf_state[layer] == 2) {
    MCFT_CUDA(cudaStreamWaitEvent(stream, c->ev_pf_done[layer], 0));
    c->pf_state[layer] = 0;
  }
  PrefetchArgs a{idx_pred, T * K, K, n_max, c->E, c->B, layer, c->policy, c->d_tag, c->d_last,
                 c->d_ins, c->d_freq, c->d_step, c->d_cnt, c->d_pfmask, c->d_pf_cancel,
                 c->d_pf_list + size_t(layer) * (1 + c->E), c->d_pf_tab + size_t(layer) * c->E,
                 c->d_slots ? c->d_slots + size_t(layer) * c->B * c->expert_bytes : nullptr,
                 c->expert_bytes, device_error_word()};
  cudaError_t e = launch_prefetch(a, stream);
  if (e != cudaSuccess) return cuda_fail(e, "prefetch kernel launch");
  if (c->d_slots) {
    MCFT_CUDA(cudaEventRecord(c->ev_pf_step[layer], stream));
    c->pf_state[layer] = 1;
  }
  return MCFT_OK;
}

mcft_status mcft_cache_prefetch_stats(const mcft_cache* c, int layer, uint64_t* prefetched,
                                      uint64_t* useful, uint64_t* bytes_moved,
                                      mcft_stream_t stream) {
  if (!c || !prefetched || !useful || !bytes_moved) return fail(MCFT_ERR_INVALID, "NULL argument");
  if (layer < -1 || layer >= c->L) return fail(MCFT_ERR_INVALID, "layer %d out of range", layer);
  std::vector<unsigned long long> h(size_t(c->L) * kCacheCounters), m(c->L);
  MCFT_CUDA(cudaMemcpyAsync(h.data(), c->d_cnt, h.size() * sizeof(h[0]), cudaMemcpyDeviceToHost, stream));
  MCFT_CUDA(cudaMemcpyAsync(m.data(), c->d_pf_moved, m.size() * sizeof(m[0]), cudaMemcpyDeviceToHost,
                            stream));
  MCFT_CUDA(cudaStreamSynchronize(stream));
  uint64_t p = 0, u = 0, b = 0;
  for (int l = 0; l < c->L; ++l) {
    if (layer >= 0 && l != layer) continue;
    p += h[size_t(l) * kCacheCounters + 3];
    u += h[size_t(l) * kCacheCounters + 4];
    b += m[l];
  }
  *prefetched = p;
  *useful = u;
  *bytes_moved = b;
  return MCFT_OK;
}

mcft_status mcft_residual_rmsnorm(const mcft_layer_desc* desc, float* x, const void* y, int T,
                                  const void* gamma, float eps, void* u, mcft_stream_t stream) {
  mcft::NvtxRange nvtx_range("mcft_residual_rmsnorm");
  mcft_status st = check_desc(desc);
  if (st != MCFT_OK) return st;
  if (T < 0) return fail(MCFT_ERR_INVALID, "T = %d < 0", T);
  if (T == 0) return MCFT_OK;
  if (!x) return fail(MCFT_ERR_INVALID, "x is NULL");
  if (gamma && !u) return fail(MCFT_ERR_INVALID, "u is NULL while gamma is given");
  if (!(eps >= 0.f) || eps > 1.f) return fail(MCFT_ERR_INVALID, "eps = %g must be in [0, 1]", eps);
  if ((reinterpret_cast<uintptr_t>(x) | reinterpret_cast<uintptr_t>(y) |
       reinterpret_cast<uintptr_t>(gamma) | reinterpret_cast<uintptr_t>(u)) & 15u)
    return fail(MCFT_ERR_INVALID, "x, y, gamma and u must be 16-byte aligned");
  NormArgs a{x, y, gamma, u, T, desc->d, eps};
  cudaError_t e = launch_resid_norm(a, desc->dtype, stream);
  if (e != cudaSuccess) return cuda_fail(e, "residual/RMSNorm kernel launch");
  return MCFT_OK;
}

mcft_status mcft_mask_sample(const float* m_tilde, const float* uniforms, int L, int E, int e_keep,
                             uint8_t* mask, float* pi, mcft_stream_t stream) {
  mcft::NvtxRange nvtx_range("mcft_mask_sample");
  if (!m_tilde || !uniforms || !mask || !pi) return fail(MCFT_ERR_INVALID, "NULL pointer argument");
  if (L < 0 || E < 1) return fail(MCFT_ERR_INVALID, "bad L = %d or E = %d", L, E);
  if (E > kMaxE) return fail(MCFT_ERR_UNSUPPORTED, "E = %d > %d", E, kMaxE);
  if (e_keep < 1 || e_keep > E)
    return fail(MCFT_ERR_INVALID, "E' = %d must be in [1, E = %d]", e_keep, E);
  if (L == 0) return MCFT_OK;
  MaskSampleArgs a{m_tilde, uniforms, L, E, e_keep, mask, pi, device_error_word()};
  cudaError_t e = launch_mask_sample(a, stream);
  if (e != cudaSuccess) return cuda_fail(e, "mask sampling kernel launch");
  return MCFT_OK;
}

mcft_status mcft_gate_grad(const mcft_layer_desc* desc, const void* dy, int T, const void* workspace,
                           size_t ws_bytes, float* dgate, mcft_stream_t stream) {
  mcft::NvtxRange nvtx_range("mcft_gate_grad");
  mcft_status st = check_desc(desc);
  if (st != MCFT_OK) return st;
  if (T < 0) return fail(MCFT_ERR_INVALID, "T = %d < 0", T);
  if (T == 0) return MCFT_OK;
  if (!dy || !workspace || !dgate) return fail(MCFT_ERR_INVALID, "NULL pointer argument");
  if (reinterpret_cast<uintptr_t>(dy) & 15u) return fail(MCFT_ERR_INVALID, "dy must be 16-byte aligned");
  const WsLayout L =
      ws_layout(desc->d, desc->E, desc->K, desc->w, desc->n_shared, desc->dtype, T);
  if (ws_bytes < L.o + size_t(L.ks) * L.mcap * desc->d * 4)
    return fail(MCFT_ERR_INVALID, "workspace of %zu bytes is not a forward workspace for T = %d",
                ws_bytes, T);
  const char* ws = static_cast<const char*>(workspace);
  GateGradArgs a{dy, reinterpret_cast<const float*>(ws + L.o), reinterpret_cast<const int*>(ws + L.pos),
                 reinterpret_cast<const WsHeader*>(ws + L.hdr), size_t(L.mcap) * desc->d, T, desc->K,
                 desc->d, L.ks, dgate};
  cudaError_t e = launch_gate_grad(a, desc->dtype, stream);
  if (e != cudaSuccess) return cuda_fail(e, "gate gradient kernel launch");
  return MCFT_OK;
}

mcft_status mcft_mask_grad(const mcft_layer_desc* desc, const int32_t* idx, const float* gate,
                           const float* dgate, int T, const float* pi, float* dm, float* dm_tilde,
                           int accumulate, mcft_stream_t stream) {
  mcft::NvtxRange nvtx_range("mcft_mask_grad");
  mcft_status st = check_desc(desc);
  if (st != MCFT_OK) return st;
  if (T < 0) return fail(MCFT_ERR_INVALID, "T = %d < 0", T);
  if (!idx || !gate || !dgate || !pi || !dm || !dm_tilde)
    return fail(MCFT_ERR_INVALID, "NULL pointer argument");
  MaskGradArgs a{idx, gate, dgate, pi, T, desc->K, desc->E, desc->gate, accumulate ? 1 : 0, dm, dm_tilde};
  cudaError_t e = launch_mask_grad(a, stream);
  if (e != cudaSuccess) return cuda_fail(e, "mask gradient kernel launch");
  return MCFT_OK;
}

mcft_status mcft_moe_forward_cached(const mcft_layer_desc* desc, const void* x, int T,
                                    const int32_t* idx, const float* gate, mcft_cache* c, int layer,
                                    const void* const* shared, void* y, void* workspace,
                                    size_t ws_bytes, mcft_stream_t compute_stream,
                                    mcft_stream_t copy_stream) {
  mcft::NvtxRange nvtx_range("mcft_moe_forward_cached");
  return mcft::forward_cached_impl(desc, x, T, idx, gate, c, layer, shared, y, workspace, ws_bytes,
                                   compute_stream, copy_stream, false);
}

}  // extern "C"

namespace mcft {

mcft_status forward_cached_impl(const mcft_layer_desc* desc, const void* x, int T,
                                const int32_t* idx, const float* gate, mcft_cache* c, int layer,
                                const void* const* shared, void* y, void* workspace,
                                size_t ws_bytes, cudaStream_t compute_stream,
                                cudaStream_t copy_stream, bool permuted) {
  mcft_status st = check_desc(desc);
  if (st != MCFT_OK) return st;
  if (!c) return fail(MCFT_ERR_INVALID, "cache is NULL");
  if (layer < 0 || layer >= c->L) return fail(MCFT_ERR_INVALID, "layer %d out of range", layer);
  if (!c->d_slots || !c->device_fetch)
    return fail(MCFT_ERR_INVALID, "the cache has no slots or its host blocks are not mapped");
  if (desc->E != c->E) return fail(MCFT_ERR_INVALID, "desc E = %d but the cache has E = %d", desc->E, c->E);
  const size_t eb = size_t(3) * desc->w * desc->d * (desc->dtype == MCFT_BF16 ? 2 : 4);
  if (eb != c->expert_bytes)
    return fail(MCFT_ERR_INVALID, "expert blocks of %zu bytes but the cache holds %zu", eb, c->expert_bytes);
  if (T < 0) return fail(MCFT_ERR_INVALID, "T = %d < 0", T);
  if (T == 0) return MCFT_OK;
  if (!x || !idx || !gate || !y || !workspace) return fail(MCFT_ERR_INVALID, "NULL pointer argument");
  const int E = desc->E, S = desc->n_shared, K = desc->K;
  if (S > 0 && !shared) return fail(MCFT_ERR_INVALID, "shared is NULL");
  for (int s = 0; s < S; ++s)
    if (!shared[s] || (reinterpret_cast<uintptr_t>(shared[s]) & 15u))
      return fail(MCFT_ERR_INVALID, "shared expert %d block is NULL or misaligned", s);
  if ((reinterpret_cast<uintptr_t>(workspace) & 255u) ||
      ((reinterpret_cast<uintptr_t>(x) | reinterpret_cast<uintptr_t>(y)) & 15u))
    return fail(MCFT_ERR_INVALID, "misaligned x, y or workspace");
  const WsLayout L = ws_layout(desc->d, E, K, desc->w, S, desc->dtype, T);
  if (L.tc)
    return fail(MCFT_ERR_UNSUPPORTED, "T = %d runs the tensor-core path; use mcft_fetch_experts + "
                "mcft_moe_forward", T);
  if (ws_bytes < L.total)
    return fail(MCFT_ERR_INVALID, "workspace of %zu bytes < %zu needed", ws_bytes, L.total);

  char* ws = static_cast<char*>(workspace);
  WsHeader* hdr = reinterpret_cast<WsHeader*>(ws + L.hdr);
  int* cnt = reinterpret_cast<int*>(ws + L.cnt);
  int* off = reinterpret_cast<int*>(ws + L.off);
  int* pos = reinterpret_cast<int*>(ws + L.pos);
  int* perm = reinterpret_cast<int*>(ws + L.perm);
  int* done = reinterpret_cast<int*>(ws + L.done);
  unsigned* err = device_error_word();
  // Small bf16 decode batches with no prefetch in flight (for any layer) fetch in the FFN's own
  // launch: its first fetch_blocks() CTAs copy the misses piece by piece and stamp each piece,
  // and the launch computes the misses with the hits, each of their items waiting for the pieces
  // it reads, so their FFN runs while the rest of the step's bytes are still on the host link and
  // no second launch waits for the copy. Otherwise a fetch kernel on the copy stream moves the
  // misses (behind this layer's prefetch, ahead of later layers') and a second FFN launch computes
  // them after it.
  int pf_any = 0;
  for (int l = 0; l < c->L; ++l) pf_any += c->pf_state[l] != 0 ? 1 : 0;
  const bool own_fetch = L.decode && T <= kStreamMaxT && c->d_landed != nullptr &&
                         c->d_fctr != nullptr && pf_any == 0;
  cudaError_t e = cudaSuccess;
  if (own_fetch) {
    if (!permuted) {
      PermuteArgs pa{idx, T, K, E, S, L.pad, L.mcap, hdr, cnt, off, pos, perm, err, done};
      e = launch_permute(pa, compute_stream);
      if (e != cudaSuccess) return cuda_fail(e, "permute kernel launch");
    }
    FfnArgs fa{};
    fa.x = x;
    fa.off = off;
    fa.perm = perm;
    fa.hdr = hdr;
    fa.done = done;
    for (int s = 0; s < S; ++s) fa.wblk[E + s] = shared[s];
    fa.h = ws + L.h;
    fa.o = reinterpret_cast<float*>(ws + L.o);
    fa.o_plane = size_t(L.mcap) * desc->d;
    fa.ksplit = L.ks;
    fa.T = T;
    fa.d = desc->d;
    fa.w = desc->w;
    fa.nseg = E + S;
    fa.E = E;
    fa.err = err;
    fa.wtab = c->d_ptr_tab + size_t(layer) * E;
    fa.ready = c->d_ready + layer;
    fa.phase = 1;  // hits, shared experts and the misses it fetches
    fa.stream = c->d_stream + layer;
    fa.fctr = c->d_fctr + 2 * size_t(layer);
    fa.landed = c->d_landed + size_t(layer) * E * c->ppe;
    fa.epoch = c->d_step + layer;
    fa.ppe = c->ppe;
    fa.fmiss = c->d_miss_dev + size_t(layer) * c->miss_stride;
    fa.fsrc = c->d_host_src + size_t(layer) * E;
    fa.fbytes = c->expert_bytes;
    fa.nfetch = fetch_blocks();
    e = launch_ffn_decode(fa, num_sms(), compute_stream, 3, 0);
    if (e != cudaSuccess) return cuda_fail(e, "expert FFN launch");
    CombineArgs ca{fa.o, gate, pos, off, hdr, y, T, desc->d, K, E, S, L.ks, fa.o_plane};
    e = launch_combine(ca, desc->dtype, compute_stream);
    if (e != cudaSuccess) return cuda_fail(e, "combine kernel launch");
    return MCFT_OK;
  }
  // 0. a prefetch of this layer decided before the step lands first (it may target the slots the
  //    step's misses overwrite)
  if (c->pf_state[layer] == 1) {
    st = enqueue_prefetch_fetches(c, copy_stream);
    if (st != MCFT_OK) return st;
  }
  // 1. the missed experts stream in on the copy stream, after this layer's cache step
  MCFT_CUDA(cudaStreamWaitEvent(copy_stream, c->ev_step[layer], 0));
  FetchArgs fe{c->d_miss_dev + size_t(layer) * c->miss_stride, c->d_host_src + size_t(layer) * E,
               c->d_ptr_tab + size_t(layer) * E, c->expert_bytes, nullptr, nullptr};
  e = launch_fetch(fe, fetch_blocks(), copy_stream);
  if (e != cudaSuccess) return cuda_fail(e, "fetch kernel launch");
  MCFT_CUDA(cudaEventRecord(c->ev_copy, copy_stream));
  // Experts a prefetch of this layer is still bringing in are not in the step's ready mask: the
  // FFN computes them in phase 2, after compute_stream waits for ev_copy, which follows their
  // fetch on this copy stream.
  if (c->pf_state[layer] == 2) c->pf_state[layer] = 0;
  // 1b. prefetches decided for later layers stream in behind this layer's misses
  int queued = 0;
  for (int l = 0; l < c->L; ++l) queued += c->pf_state[l] == 1 ? 1 : 0;
  st = enqueue_prefetch_fetches(c, copy_stream);
  if (st != MCFT_OK) return st;
  // 2. meanwhile: permutation (unless the fused prologue wrote it into this workspace) and the
  //    experts that were hits (and the shared experts)
  if (!permuted) {
    PermuteArgs pa{idx, T, K, E, S, L.pad, L.mcap, hdr, cnt, off, pos, perm, err, done};
    e = launch_permute(pa, compute_stream);
    if (e != cudaSuccess) return cuda_fail(e, "permute kernel launch");
  }
  FfnArgs fa{};
  fa.x = x;
  fa.off = off;
  fa.perm = perm;
  fa.hdr = hdr;
  fa.done = done;  // fused decode FFN (claimed items)
  for (int s = 0; s < S; ++s) fa.wblk[E + s] = shared[s];
  fa.h = ws + L.h;
  fa.o = reinterpret_cast<float*>(ws + L.o);
  fa.o_plane = size_t(L.mcap) * desc->d;
  fa.ksplit = L.ks;
  fa.T = T;
  fa.d = desc->d;
  fa.w = desc->w;
  fa.nseg = E + S;
  fa.E = E;
  fa.err = err;
  fa.wtab = c->d_ptr_tab + size_t(layer) * E;
  fa.ready = c->d_ready + layer;
  // A fetch kernel running alongside keeps its SM slots: this layer's misses (or an earlier
  // prefetch still on the copy stream) during phase 1; during phase 2, which starts after the
  // misses have landed, only prefetches queued behind them at 1b.
  for (int phase = 1; phase <= 2; ++phase) {
    fa.phase = phase;
    if (phase == 2) MCFT_CUDA(cudaStreamWaitEvent(compute_stream, c->ev_copy, 0));
    const int reserved = phase == 1 || queued > 0 ? fetch_blocks() : 0;
    e = L.decode ? launch_ffn_decode(fa, num_sms(), compute_stream, 3, reserved)
                 : launch_ffn_rowwise(fa, desc->dtype, num_sms(), compute_stream);
    if (e != cudaSuccess) return cuda_fail(e, "expert FFN launch");
  }
  CombineArgs ca{fa.o, gate, pos, off, hdr, y, T, desc->d, K, E, S, L.ks, fa.o_plane};
  e = launch_combine(ca, desc->dtype, compute_stream);
  if (e != cudaSuccess) return cuda_fail(e, "combine kernel launch");
  return MCFT_OK;
}

mcft_status stack_prologue(const mcft_layer_desc* desc, float* x, const void* y, const void* gamma,
                           const void* gamma_next, float eps, void* u, const void* w_router,
                           const float* prior, int32_t* idx, float* gate, const void* w_router_next,
                           const float* prior_next, int32_t* pred, float* gate_pred,
                           mcft_cache* c, int layer, int n_prefetch, void* workspace,
                           size_t ws_bytes, cudaStream_t stream) {
  const int E = desc->E, K = desc->K, S = desc->n_shared;
  if (!prologue_supported(desc->d, E, 1) || K > kMaxK)
    return fail(MCFT_ERR_UNSUPPORTED, "the fused prologue serves one token with d <= 4096, K <= 8");
  if (layer < 0 || layer >= c->L) return fail(MCFT_ERR_INVALID, "layer %d out of range", layer);
  const bool do_pred = gamma_next != nullptr;
  const bool do_pf = do_pred && n_prefetch > 0 && layer + 1 < c->L;
  if (do_pf && (n_prefetch > c->B || (c->d_slots && !c->device_fetch)))
    return fail(MCFT_ERR_INVALID, "bad prefetch settings");
  const WsLayout L = ws_layout(desc->d, E, K, desc->w, S, desc->dtype, 1);
  if (ws_bytes < L.total) return fail(MCFT_ERR_INVALID, "workspace too small");
  if (do_pf) {
    if (c->pf_state[layer + 1] == 1)
      return fail(MCFT_ERR_INVALID, "the previous prefetch of layer %d was never fetched", layer + 1);
    if (c->pf_state[layer + 1] == 2) {
      MCFT_CUDA(cudaStreamWaitEvent(stream, c->ev_pf_done[layer + 1], 0));
      c->pf_state[layer + 1] = 0;
    }
  }
  unsigned* err = device_error_word();
  PrologueArgs a{};
  a.x = x;
  a.y = y;
  a.gamma = gamma;
  a.gamma_next = gamma_next;
  a.u = u;
  a.eps = eps;
  a.d = desc->d;
  auto route_args = [&](RouteArgs& r, const void* w, const float* pri, int32_t* out, float* g) {
    r.x = u;
    r.w_router = w;
    r.T = 1;
    r.d = desc->d;
    r.E = E;
    r.K = K;
    r.mode = MCFT_ROUTE_SOFT_PRIOR;
    r.gate_mode = desc->gate;
    for (int e = 0; e < E; ++e) r.prior[e] = pri[e];
    r.idx = out;
    r.gate = g;
    r.err = err;
  };
  route_args(a.route, w_router, prior, idx, gate);
  if (do_pred) route_args(a.pred, w_router_next, prior_next, pred, gate_pred);
  a.cache = CacheStepArgs{idx, K, E, c->B, layer, c->policy, c->d_tag, c->d_last, c->d_ins,
                          c->d_freq, c->d_step, c->d_cnt, c->d_pfmask, c->d_pf_cancel,
                          c->d_miss + size_t(layer) * c->miss_stride,
                          c->d_miss_dev + size_t(layer) * c->miss_stride,
                          c->d_ptr_tab + size_t(layer) * E, c->d_ready + layer, c->d_stream + layer,
                          c->d_fctr ? c->d_fctr + 2 * size_t(layer) : nullptr,
                          c->d_slots ? c->d_slots + size_t(layer) * c->B * c->expert_bytes : nullptr,
                          c->d_staging, c->expert_bytes, err};
  a.do_prefetch = do_pf ? 1 : 0;
  if (do_pf) {
    const int l1 = layer + 1;
    a.prefetch = PrefetchArgs{pred, K, K, n_prefetch, E, c->B, l1, c->policy, c->d_tag, c->d_last,
                              c->d_ins, c->d_freq, c->d_step, c->d_cnt, c->d_pfmask, c->d_pf_cancel,
                              c->d_pf_list + size_t(l1) * (1 + E), c->d_pf_tab + size_t(l1) * E,
                              c->d_slots ? c->d_slots + size_t(l1) * c->B * c->expert_bytes : nullptr,
                              c->expert_bytes, err};
  }
  char* ws = static_cast<char*>(workspace);
  a.perm = PermuteArgs{idx, 1, K, E, S, L.pad, L.mcap, reinterpret_cast<WsHeader*>(ws + L.hdr),
                       reinterpret_cast<int*>(ws + L.cnt), reinterpret_cast<int*>(ws + L.off),
                       reinterpret_cast<int*>(ws + L.pos), reinterpret_cast<int*>(ws + L.perm), err,
                       reinterpret_cast<int*>(ws + L.done)};
  cudaError_t e = launch_prologue(a, desc->dtype, stream);
  if (e != cudaSuccess) return cuda_fail(e, "prologue kernel launch");
  MCFT_CUDA(cudaEventRecord(c->ev_step[layer], stream));
  if (do_pf && c->d_slots) {
    MCFT_CUDA(cudaEventRecord(c->ev_pf_step[layer + 1], stream));
    c->pf_state[layer + 1] = 1;
  }
  return MCFT_OK;
}

}  // namespace mcft

extern "C" {

mcft_status mcft_cache_last_misses(const mcft_cache* c, int layer, int* n_out, int32_t* experts,
                                   int32_t* slots) {
  if (!c || !n_out || !experts || !slots) return fail(MCFT_ERR_INVALID, "NULL argument");
  if (layer < 0 || layer >= c->L) return fail(MCFT_ERR_INVALID, "layer %d out of range", layer);
  const int32_t* m = c->h_miss + size_t(layer) * c->miss_stride;
  const int nm = m[0];
  if (nm < 0 || nm > c->E) return fail(MCFT_ERR_INVALID, "corrupt miss list");
  *n_out = nm;
  for (int i = 0; i < nm; ++i) {
    experts[i] = m[1 + i];
    slots[i] = m[1 + c->E + i];
  }
  return MCFT_OK;
}

mcft_status mcft_cache_stats(const mcft_cache* c, int layer, uint64_t* hits, uint64_t* fetches,
                             uint64_t* bypass, mcft_stream_t stream) {
  if (!c || !hits || !fetches || !bypass) return fail(MCFT_ERR_INVALID, "NULL argument");
  if (layer < -1 || layer >= c->L) return fail(MCFT_ERR_INVALID, "layer %d out of range", layer);
  std::vector<unsigned long long> h(size_t(c->L) * kCacheCounters);
  MCFT_CUDA(cudaMemcpyAsync(h.data(), c->d_cnt, h.size() * sizeof(h[0]), cudaMemcpyDeviceToHost, stream));
  MCFT_CUDA(cudaStreamSynchronize(stream));
  uint64_t a = 0, b = 0, d = 0;
  for (int l = 0; l < c->L; ++l) {
    if (layer >= 0 && l != layer) continue;
    a += h[size_t(l) * kCacheCounters];
    b += h[size_t(l) * kCacheCounters + 1];
    d += h[size_t(l) * kCacheCounters + 2];
  }
  *hits = a;
  *fetches = b;
  *bypass = d;
  return MCFT_OK;
}

mcft_status mcft_cache_tags(const mcft_cache* c, int layer, int32_t* tags, mcft_stream_t stream) {
  if (!c || !tags) return fail(MCFT_ERR_INVALID, "NULL argument");
  if (layer < 0 || layer >= c->L) return fail(MCFT_ERR_INVALID, "layer %d out of range", layer);
  MCFT_CUDA(cudaMemcpyAsync(tags, c->d_tag + size_t(layer) * c->B, sizeof(int32_t) * c->B,
                            cudaMemcpyDeviceToHost, stream));
  MCFT_CUDA(cudaStreamSynchronize(stream));
  return MCFT_OK;
}

mcft_status mcft_cache_export(const mcft_cache* c, void* buf, size_t* bytes, mcft_stream_t stream) {
  if (!c || !bytes) return fail(MCFT_ERR_INVALID, "NULL argument");
  const size_t LB = size_t(c->L) * c->B, LE = size_t(c->L) * c->E;
  const size_t need = state_bytes(c);
  if (!buf) {
    *bytes = need;
    return MCFT_OK;
  }
  if (*bytes < need) return fail(MCFT_ERR_INVALID, "buffer of %zu bytes < %zu needed", *bytes, need);
  char* p = static_cast<char*>(buf);
  CacheStateHeader h{kStateMagic, uint32_t(c->L), uint32_t(c->E), uint32_t(c->B), uint32_t(c->policy), 0};
  memcpy(p, &h, sizeof(h));
  p += sizeof(h);
  const struct { const void* src; size_t n; } parts[] = {
      {c->d_tag, LB * 4}, {c->d_last, LB * 8}, {c->d_ins, LB * 8}, {c->d_freq, LE * 8},
      {c->d_step, size_t(c->L) * 8}, {c->d_cnt, size_t(c->L) * 8 * kCacheCounters},
      {c->d_pfmask, size_t(c->L) * 8}};
  for (const auto& part : parts) {
    MCFT_CUDA(cudaMemcpyAsync(p, part.src, part.n, cudaMemcpyDeviceToHost, stream));
    p += part.n;
  }
  MCFT_CUDA(cudaStreamSynchronize(stream));
  *bytes = need;
  return MCFT_OK;
}

mcft_status mcft_cache_import(mcft_cache* c, const void* buf, size_t bytes, mcft_stream_t stream) {
  if (!c || !buf) return fail(MCFT_ERR_INVALID, "NULL argument");
  const size_t LB = size_t(c->L) * c->B, LE = size_t(c->L) * c->E;
  const size_t need = state_bytes(c);
  if (bytes < need) return fail(MCFT_ERR_INVALID, "state of %zu bytes < %zu expected", bytes, need);
  const char* p = static_cast<const char*>(buf);
  CacheStateHeader h;
  memcpy(&h, p, sizeof(h));
  if (h.magic != kStateMagic || h.L != uint32_t(c->L) || h.E != uint32_t(c->E) ||
      h.B != uint32_t(c->B) || h.policy != uint32_t(c->policy))
    return fail(MCFT_ERR_INVALID, "state was exported from a cache of another shape or policy");
  p += sizeof(h);
  const int32_t* tags = reinterpret_cast<const int32_t*>(p);
  for (size_t i = 0; i < LB; ++i)
    if (tags[i] < -1 || tags[i] >= c->E) return fail(MCFT_ERR_INVALID, "corrupt tag in state");
  const struct { void* dst; size_t n; } parts[] = {
      {c->d_tag, LB * 4}, {c->d_last, LB * 8}, {c->d_ins, LB * 8}, {c->d_freq, LE * 8},
      {c->d_step, size_t(c->L) * 8}, {c->d_cnt, size_t(c->L) * 8 * kCacheCounters},
      {c->d_pfmask, size_t(c->L) * 8}};
  for (const auto& part : parts) {
    MCFT_CUDA(cudaMemcpyAsync(part.dst, p, part.n, cudaMemcpyHostToDevice, stream));
    p += part.n;
  }
  // landed stamps may carry the epochs of steps taken after the exported state: clear them
  if (c->d_landed)
    MCFT_CUDA(cudaMemsetAsync(c->d_landed, 0, sizeof(unsigned) * size_t(c->L) * c->E * c->ppe, stream));
  MCFT_CUDA(cudaStreamSynchronize(stream));
  return MCFT_OK;
}

void mcft_cache_destroy(mcft_cache* c) {
  if (!c) return;
  cudaDeviceSynchronize();
  cache_free(c);
}

}  // extern "C"
