// hs_static.cu -- hs_feedback_static: hs_feedback without a caller-supplied
// workspace.  Its scratch is a fixed array in the library's device image,
// so the call allocates nothing on any path.
#include <cuda.h>  // CUcontext / CUresult types; the functions come from the runtime
#include <cuda_runtime.h>

#include <mutex>

#include "hedgefb.h"

namespace {

// Scratch of every hs_feedback_static call on a device.  Each GPU that loads
// the library holds these bytes until the process exits.
static __device__ __align__(256) unsigned char g_static_scratch[HS_STATIC_SCRATCH_BYTES];

constexpr int kMaxDevices = 64;

// Device address of g_static_scratch per device, found by the first call
// made with that device current, together with the id of the context it
// belongs to.  In host code the array's own name is only a host-side
// stand-in, never a device address.  A device reset (or anything else that
// replaces the context) gives the device a new context id, and the next
// call looks the address up again instead of using a stale one.
struct Entry {
  bool valid;
  unsigned long long ctx_id;
  void* addr;
};
std::mutex g_mu;
Entry g_entry[kMaxDevices];

using CtxGetCurrentFn = CUresult (*)(CUcontext*);
using CtxGetIdFn = CUresult (*)(CUcontext, unsigned long long*);

// The process-unique id of the context current on this thread; false when
// there is none yet (or the driver lacks the query).
bool current_context_id(unsigned long long* id) {
  static CtxGetCurrentFn get_current = nullptr;
  static CtxGetIdFn get_id = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* f = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &f, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      get_current = reinterpret_cast<CtxGetCurrentFn>(f);
    f = nullptr;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetId", &f, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      get_id = reinterpret_cast<CtxGetIdFn>(f);
  });
  if (!get_current || !get_id) return false;
  CUcontext ctx = nullptr;
  if (get_current(&ctx) != CUDA_SUCCESS || !ctx) return false;
  return get_id(ctx, id) == CUDA_SUCCESS;
}

// The scratch's device address in the current device's current context.
hs_status scratch_address(void** out) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return HS_ERR_CUDA;
  if (dev < 0 || dev >= kMaxDevices) return HS_ERR_UNSUPPORTED;
  std::lock_guard<std::mutex> lock(g_mu);
  Entry& e = g_entry[dev];
  unsigned long long id = 0;
  if (e.valid && current_context_id(&id) && id == e.ctx_id) {
    *out = e.addr;
    return HS_OK;
  }
  // set-up for this device and context (it also creates the device's
  // primary context if no runtime call has yet)
  void* addr = nullptr;
  if (cudaGetSymbolAddress(&addr, g_static_scratch) != cudaSuccess || !addr) return HS_ERR_CUDA;
  if (!current_context_id(&id)) return HS_ERR_CUDA;
  e.valid = true;
  e.ctx_id = id;
  e.addr = addr;
  *out = addr;
  return HS_OK;
}

}  // namespace

extern "C" hs_status hs_feedback_static(const void* target, const void* drafter, int dtype, int N,
                                        int B, int P, int V, float temperature, int greedy,
                                        float* alpha, float* e_len, int* dev_status,
                                        void* stream) {
  const size_t need = hs_feedback_workspace_size(N, B, P, V, dtype, greedy);
  if (need > HS_STATIC_SCRATCH_BYTES) return HS_ERR_UNSUPPORTED;
  void* scratch = nullptr;
  const hs_status st = scratch_address(&scratch);
  if (st != HS_OK) return st;
  return hs_feedback(target, drafter, dtype, N, B, P, V, temperature, greedy, alpha, e_len,
                     scratch, HS_STATIC_SCRATCH_BYTES, dev_status, stream);
}
