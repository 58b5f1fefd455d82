// Rotate-quantize kernel variants for __half input.
#include "rq_launch.cuh"

namespace clq {

cudaError_t launch_rotate_quant_f16(const RotateQuantArgs& a, int logb, int threads, size_t smem,
                                   int sms, cudaStream_t st) {
  return rq::launch_rotate_quant_t<__half>(a, logb, threads, smem, sms, st);
}

}  // namespace clq
