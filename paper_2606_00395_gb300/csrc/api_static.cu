// pr2_moe_forward_static: the layer forward of pr2_moe_forward for callers that cannot hand the
// library a workspace buffer.
//
// Some callers cannot allocate device memory at the point where they run the layer: a runtime
// that owns every byte of device memory through its own pool and has no spare block to lend, a
// host environment that forbids device allocation on its hot path (cudaMalloc and cudaFree can
// synchronise the whole device), or a plug-in whose memory budget is fixed when it is loaded.
// For them this entry point takes its scratch from one array compiled into this library
// (kStaticScratchBytes, reserved on every GPU that loads the library until the process exits),
// so the call allocates nothing.
#include <mutex>

#include "pr2_internal.h"

namespace pr2 {
namespace {

constexpr size_t kStaticScratchBytes = size_t{32} << 20;  // 32 MiB
constexpr int kMaxDevices = 64;

// File-scope scratch shared by every call of pr2_moe_forward_static on a device.
static __device__ __align__(256) uint8_t pr2_static_scratch[kStaticScratchBytes];

std::mutex g_scratch_mutex;
void* g_scratch_ptr[kMaxDevices] = {};

// Device address of the scratch array on the current device.  In host code the array's name
// is only a host-side stand-in, so the address comes from cudaGetSymbolAddress, looked up once
// per device with that device current.
pr2_status static_scratch(void** out) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return PR2_ERR_CUDA;
  if (dev < 0 || dev >= kMaxDevices) return PR2_ERR_UNSUPPORTED;
  std::lock_guard<std::mutex> lock(g_scratch_mutex);
  if (g_scratch_ptr[dev] == nullptr) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, pr2_static_scratch) != cudaSuccess || p == nullptr)
      return PR2_ERR_CUDA;
    g_scratch_ptr[dev] = p;
  }
  *out = g_scratch_ptr[dev];
  return PR2_OK;
}

}  // namespace
}  // namespace pr2

extern "C" {

size_t pr2_static_scratch_bytes(void) { return pr2::kStaticScratchBytes; }

pr2_status pr2_moe_forward_static(const pr2_dims* dims, const void* h, const int32_t* idx,
                                  const float* gates, const void* W_gate, const void* W_up,
                                  const void* W_down, const void* Ws_gate, const void* Ws_up,
                                  const void* Ws_down, void* out, int32_t* counts,
                                  int32_t* perm, int32_t* status_dev, void* stream) {
  const size_t need = pr2_moe_workspace_bytes(dims);
  if (need == 0) return PR2_ERR_INVALID_ARG;
  if (need > pr2::kStaticScratchBytes) return PR2_ERR_WORKSPACE;  // layer too large
  void* scratch = nullptr;
  const pr2_status s = pr2::static_scratch(&scratch);
  if (s != PR2_OK) return s;
  // pr2_moe_forward clears the scratch status word itself when status_dev is NULL; every other
  // scratch region is fully written before it is read, so nothing else needs zeroing.
  return pr2_moe_forward(dims, h, idx, gates, W_gate, W_up, W_down, Ws_gate, Ws_up, Ws_down, out,
                         counts, perm, scratch, pr2::kStaticScratchBytes, status_dev, nullptr,
                         stream);
}

}  // extern "C"
