// Hot-path rotate-quantize kernel variants (paired-row loop for b = 32, wide
// segments for b >= 64): __half input, E2M3 codes.
#include "rq_launch.cuh"

namespace clq {

cudaError_t launch_rotate_quant_pair_f16_e2m3(const RotateQuantArgs& a, int logb, int half,
                                              int threads, size_t smem, int sms,
                                              cudaStream_t st) {
  return rq::launch_rotate_quant_pair_t<__half, 3>(a, logb, half, threads, smem, sms, st);
}

cudaError_t launch_rotate_quant_wide_f16_e2m3(const RotateQuantArgs& a, int logb, int stage,
                                              int threads, size_t smem, int sms,
                                              cudaStream_t st) {
  return rq::launch_rotate_quant_wide_t<__half, 3>(a, logb, stage, threads, smem, sms, st);
}

}  // namespace clq
