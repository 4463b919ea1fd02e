// mcft_moe_forward_noalloc: the expert FFN + combine of mcft_moe_forward for callers that cannot
// allocate device memory themselves, using a fixed scratch array that lives in the library.
//
// Some callers may not call cudaMalloc (or any allocator) at the point where they run a layer:
// a plugin embedded in an application that owns every device allocation through its own pool, or
// a latency-critical decode loop where an allocation's implicit device synchronisation is not
// acceptable. They still own x, idx, gate, the expert blocks and y; only the scratch space that
// mcft_moe_forward takes as `workspace` comes from here instead.
//
// The scratch is one file-scope device array of kScratchBytes (16 MiB), 256-byte aligned. Every
// GPU that loads the library holds it until the process exits. It is large enough for the decode
// shapes (up to 64 tokens per call for the Mixtral- and DeepSeek-V2-Lite-shaped layers); larger
// calls are rejected with MCFT_ERR_UNSUPPORTED. In host code the array's name is only a host-side
// stand-in, so the device address is looked up once per device with cudaGetSymbolAddress, with
// that device current, on the first call made on it (make that first call before any stream
// capture). The looked-up address is kept for the life of the process: after a cudaDeviceReset
// the context it belonged to is gone, and this entry point must not be called on that device
// again. Every call shares the array and it keeps the last call's contents: nothing in it needs
// to start at zero (the first kernel of a call writes the header and offsets the later kernels
// read), but calls whose kernels overlap on the GPU (different streams, or different host threads)
// race on it and must be serialised by the caller. This entry point calls no cudaMalloc,
// cudaFree or other allocating routine (with kernel timing off, the default).
#include <cuda_runtime.h>
#include <stdio.h>

#include <mutex>

#include "common.cuh"
#include "internal.h"

// The scratch array (file scope, internal linkage).
static constexpr size_t kScratchBytes = size_t(16) << 20;
static __device__ __align__(256) unsigned char g_noalloc_scratch[kScratchBytes];

namespace mcft {
namespace {

constexpr int kMaxDevicesNoAlloc = 64;

std::mutex g_scratch_mu;
void* g_scratch_addr[kMaxDevicesNoAlloc] = {nullptr};

// Device address of the scratch array on the current device (looked up once per device).
mcft_status scratch_address(void** out) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return set_error_message(MCFT_ERR_CUDA, cudaGetErrorString(e));
  if (dev < 0 || dev >= kMaxDevicesNoAlloc)
    return set_error_message(MCFT_ERR_UNSUPPORTED, "device index beyond the scratch table");
  std::lock_guard<std::mutex> lock(g_scratch_mu);
  if (!g_scratch_addr[dev]) {
    void* p = nullptr;
    e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
    if (e != cudaSuccess || !p)
      return set_error_message(MCFT_ERR_CUDA, "cudaGetSymbolAddress of the scratch array failed");
    g_scratch_addr[dev] = p;
  }
  *out = g_scratch_addr[dev];
  return MCFT_OK;
}

}  // namespace
}  // namespace mcft

using namespace mcft;

extern "C" mcft_status mcft_moe_forward_noalloc(const mcft_layer_desc* desc, const void* x, int T,
                                                const int32_t* idx, const float* gate,
                                                const void* const* experts,
                                                const void* const* shared, void* y,
                                                mcft_stream_t stream) {
  mcft::NvtxRange nvtx_range("mcft_moe_forward_noalloc");
  size_t need = 0;
  mcft_status st = mcft_moe_workspace_size(desc, T, &need);
  if (st != MCFT_OK) return st;
  if (need > kScratchBytes) {
    char msg[256];
    snprintf(msg, sizeof(msg),
             "this call needs %zu bytes of scratch, more than the %zu-byte static array of "
             "mcft_moe_forward_noalloc; use mcft_moe_forward with a workspace",
             need, kScratchBytes);
    return set_error_message(MCFT_ERR_UNSUPPORTED, msg);
  }
  void* scratch = nullptr;
  st = scratch_address(&scratch);
  if (st != MCFT_OK) return st;
  return mcft_moe_forward(desc, x, T, idx, gate, experts, shared, y, scratch, kScratchBytes, stream);
}
