// Rotate-quantize kernel variants for __nv_bfloat16 input.
#include "rq_launch.cuh"

namespace clq {

cudaError_t launch_rotate_quant_bf16(const RotateQuantArgs& a, int logb, int threads, size_t smem,
                                   int sms, cudaStream_t st) {
  return rq::launch_rotate_quant_t<__nv_bfloat16>(a, logb, threads, smem, sms, st);
}

}  // namespace clq
