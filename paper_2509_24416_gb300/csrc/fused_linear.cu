// Fused rotate-quant + W4A4 GEMM (placeholder until the fused kernel lands).
#include "clq_device.cuh"
#include "clq_kernels.h"

namespace clq {

cudaError_t launch_fused_linear(const uint8_t*, const FusedArgs&, int, cudaStream_t) {
  return cudaErrorNotSupported;
}

}  // namespace clq
