// hs_static.cu -- hs_feedback_static: hs_feedback without a caller-supplied
// workspace.  Its scratch is a fixed array in the library's device image,
// so the call allocates nothing on any path.
#include <cuda_runtime.h>

#include <atomic>

#include "hedgefb.h"

namespace {

// Scratch of every hs_feedback_static call on a device.  Each GPU that loads
// the library holds these bytes until the process exits.
static __device__ __align__(256) unsigned char g_static_scratch[HS_STATIC_SCRATCH_BYTES];

constexpr int kMaxDevices = 64;
// Device address of g_static_scratch per device, found on the first call
// made with that device current.  In host code the array's own name is only
// a host-side stand-in, never a device address.
std::atomic<void*> g_scratch_addr[kMaxDevices];

}  // namespace

extern "C" hs_status hs_feedback_static(const void* target, const void* drafter, int dtype, int N,
                                        int B, int P, int V, float temperature, int greedy,
                                        float* alpha, float* e_len, int* dev_status,
                                        void* stream) {
  const size_t need = hs_feedback_workspace_size(N, B, P, V, dtype, greedy);
  if (need > HS_STATIC_SCRATCH_BYTES) return HS_ERR_UNSUPPORTED;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return HS_ERR_CUDA;
  if (dev < 0 || dev >= kMaxDevices) return HS_ERR_UNSUPPORTED;
  void* scratch = g_scratch_addr[dev].load(std::memory_order_acquire);
  if (!scratch) {
    if (cudaGetSymbolAddress(&scratch, g_static_scratch) != cudaSuccess || !scratch)
      return HS_ERR_CUDA;
    g_scratch_addr[dev].store(scratch, std::memory_order_release);
  }
  return hs_feedback(target, drafter, dtype, N, B, P, V, temperature, greedy, alpha, e_len,
                     scratch, HS_STATIC_SCRATCH_BYTES, dev_status, stream);
}
