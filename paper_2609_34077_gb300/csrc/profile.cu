// Kernel timing: when enabled, every launch site of the library brackets its kernel with a pair of
// CUDA events on the launching stream; totals per kernel are read back (after synchronising the
// recorded events) through mcft_profile_read. Off by default, so calls record nothing.
#include <cuda_runtime.h>

#include <atomic>
#include <mutex>
#include <vector>

#include "internal.h"

namespace mcft {
namespace {

const char* const kNames[kProfCount] = {
    "route",     "cache_step", "permute", "gather",       "ffn13_rowwise", "ffn2_rowwise",
    "gemm13_tc", "gemm2_tc",   "combine", "ffn13_decode", "ffn2_decode", "fetch", "lora_down",
    "rmsnorm",   "prefetch",   "fetch_prefetch", "prologue", "ffn_decode", "host_copy",
    "ffn_decode_fetch", "gemm13_tc_pair", "gemm2_tc_pair"};

struct Pending {
  int kid;
  cudaEvent_t start, stop;
};

std::atomic<bool> g_enabled{false};
std::mutex g_mu;
std::vector<Pending> g_pending;
std::vector<cudaEvent_t> g_free;
uint64_t g_launches[kProfCount];
double g_ms[kProfCount];
Pending g_open[kProfCount];
bool g_is_open[kProfCount];

cudaEvent_t take_event() {
  if (!g_free.empty()) {
    cudaEvent_t e = g_free.back();
    g_free.pop_back();
    return e;
  }
  cudaEvent_t e = nullptr;
  cudaEventCreate(&e);
  return e;
}

void drain_locked() {
  for (Pending& p : g_pending) {
    float ms = 0.f;
    if (cudaEventSynchronize(p.stop) == cudaSuccess && cudaEventElapsedTime(&ms, p.start, p.stop) == cudaSuccess) {
      g_launches[p.kid] += 1;
      g_ms[p.kid] += ms;
    }
    g_free.push_back(p.start);
    g_free.push_back(p.stop);
  }
  g_pending.clear();
}

}  // namespace

void prof_begin(int kid, cudaStream_t s) {
  if (!g_enabled.load(std::memory_order_relaxed)) return;
  std::lock_guard<std::mutex> lock(g_mu);
  Pending p{kid, take_event(), take_event()};
  cudaEventRecord(p.start, s);
  g_open[kid] = p;
  g_is_open[kid] = true;
}

void prof_end(int kid, cudaStream_t s) {
  if (!g_enabled.load(std::memory_order_relaxed)) return;
  std::lock_guard<std::mutex> lock(g_mu);
  if (!g_is_open[kid]) return;
  g_is_open[kid] = false;
  cudaEventRecord(g_open[kid].stop, s);
  g_pending.push_back(g_open[kid]);
}

}  // namespace mcft

using namespace mcft;

extern "C" {

mcft_status mcft_profile_enable(int on) {
  g_enabled.store(on != 0);
  return MCFT_OK;
}

mcft_status mcft_profile_reset(void) {
  std::lock_guard<std::mutex> lock(g_mu);
  drain_locked();
  for (int i = 0; i < kProfCount; ++i) {
    g_launches[i] = 0;
    g_ms[i] = 0.0;
  }
  return MCFT_OK;
}

mcft_status mcft_profile_read(int max, const char** names, uint64_t* launches, double* ms, int* n_out) {
  if (!n_out || (max > 0 && (!names || !launches || !ms))) return MCFT_ERR_INVALID;
  std::lock_guard<std::mutex> lock(g_mu);
  drain_locked();
  const int n = max < kProfCount ? max : kProfCount;
  for (int i = 0; i < n; ++i) {
    names[i] = kNames[i];
    launches[i] = g_launches[i];
    ms[i] = g_ms[i];
  }
  *n_out = kProfCount;
  return MCFT_OK;
}

}  // extern "C"
