// saki_score_topk_noalloc: saki_score_topk with a static device scratch array
// instead of a caller-provided workspace, for callers that cannot allocate
// device memory (see include/saki.h).  No cudaMalloc / cudaFree anywhere.
#include <atomic>

#include "common.cuh"
#include "kernels.h"

// The scratch.  On the host this name is only a stand-in for the device array
// (passing it to a kernel would fault, or read host memory where the GPU can
// reach it): host code uses the address cudaGetSymbolAddress returns.
static __device__ __align__(256) unsigned char g_noalloc_scratch[SAKI_NOALLOC_SCRATCH_BYTES];

namespace {
constexpr int kMaxDevices = 64;
std::atomic<void*> g_scratch_addr[kMaxDevices];  // device address per device ordinal

// The scratch's device address on the current device, looked up on first use.
saki_status scratch_addr(void** out) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return SAKI_ERR_CUDA;
  if (dev < 0 || dev >= kMaxDevices) return SAKI_ERR_UNSUPPORTED;
  void* addr = g_scratch_addr[dev].load(std::memory_order_acquire);
  if (!addr) {  // once per device, with that device current
    if (cudaGetSymbolAddress(&addr, g_noalloc_scratch) != cudaSuccess) return SAKI_ERR_CUDA;
    g_scratch_addr[dev].store(addr, std::memory_order_release);
  }
  *out = addr;
  return SAKI_OK;
}
}  // namespace

extern "C" saki_status saki_noalloc_status(saki_stream stream) {
  void* addr = nullptr;
  const saki_status st = scratch_addr(&addr);
  if (st != SAKI_OK) return st;
  saki::PageableUploads pageable;
  return saki_workspace_status(addr, stream);
}

extern "C" saki_status saki_score_topk_noalloc(const saki_config* cfg, const saki_layout* layout, const void* Q,
                                               const float* L, const void* sketch, const float* nu, int32_t* idx,
                                               float* score, saki_stream stream) {
  void* addr = nullptr;
  const saki_status st = scratch_addr(&addr);
  if (st != SAKI_OK) return st;
  saki::PageableUploads pageable;   // no pinned staging either: its first use allocates
  return saki_score_topk(cfg, layout, Q, L, sketch, nu, idx, score, addr, SAKI_NOALLOC_SCRATCH_BYTES, stream);
}
