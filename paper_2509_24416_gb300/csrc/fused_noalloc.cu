// clq_fused_linear_noalloc: the fused linear layer for callers that cannot
// allocate device memory when they run it (plugin enqueue hooks of inference
// engines, serving loops that forbid allocation after start-up, code without
// an allocator handle).  Instead of a caller-provided workspace it uses one
// scratch array defined here in static device memory, so the call allocates
// and frees nothing; it forwards to clq_fused_linear with that array.
#include <atomic>

#include <cuda_runtime.h>

#include "../../include/clq.h"
#include "clq_kernels.h"

namespace {

// The scratch array.  Every device that loads the library holds it until the
// process exits.  Host code must not pass `g_noalloc_scratch` itself to a
// kernel (on the host it names a stand-in, not a device address); the device
// address comes from cudaGetSymbolAddress below.
__device__ __align__(256) unsigned char g_noalloc_scratch[CLQ_NOALLOC_SCRATCH_BYTES];

constexpr int kMaxDevices = 64;
std::atomic<void*> g_scratch_ptr[kMaxDevices];

// Device address of the scratch array on the current device, resolved on the
// first call for that device (which is why that call should come before any
// stream capture).
clq_status scratch_address(void** out) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return CLQ_ERR_CUDA;
  if (dev < 0 || dev >= kMaxDevices) return CLQ_ERR_UNSUPPORTED;
  void* p = g_scratch_ptr[dev].load(std::memory_order_acquire);
  if (p == nullptr) {
    void* q = nullptr;
    if (cudaGetSymbolAddress(&q, g_noalloc_scratch) != cudaSuccess || q == nullptr) {
      cudaGetLastError();  // leave no error behind for the caller's next check
      return CLQ_ERR_CUDA;
    }
    g_scratch_ptr[dev].store(q, std::memory_order_release);
    p = q;
  }
  *out = p;
  return CLQ_OK;
}

}  // namespace

extern "C" clq_status clq_fused_linear_noalloc(const void* X, clq_dtype dtype, int32_t M,
                                               int32_t K, int32_t ldx, const int32_t* perm,
                                               int32_t b, const uint8_t* W,
                                               clq_codes w_codes, const float* s_w,
                                               const void* bias, int32_t N, void* Y,
                                               void* stream) {
  // The same checks, in the same order, as clq_fused_linear; an empty problem
  // is a no-op whatever its size.
  bool noop = false;
  clq_status st = clq::fused_linear_check(X, dtype, M, K, ldx, perm, b, W, w_codes, s_w, bias,
                                          N, Y, &noop);
  if (st != CLQ_OK || noop) return st;
  if (clq_fused_linear_workspace_size(M, K) > CLQ_NOALLOC_SCRATCH_BYTES)
    return CLQ_ERR_SCRATCH_LIMIT;
  // An unsupported device is reported as such before the symbol is looked up.
  st = clq::device_check();
  if (st != CLQ_OK) return st;
  void* scratch = nullptr;
  st = scratch_address(&scratch);
  if (st != CLQ_OK) return st;
  // The forwarded call clears the counters it needs in the scratch array and
  // launches on `stream`.
  return clq_fused_linear(X, dtype, M, K, ldx, perm, b, W, w_codes, s_w, bias, N, Y, scratch,
                          CLQ_NOALLOC_SCRATCH_BYTES, stream);
}
