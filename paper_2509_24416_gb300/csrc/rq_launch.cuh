// Standalone rotate-quantize kernel and its launch templates, instantiated
// once per input type (rotate_quant_f16.cu, rotate_quant_bf16.cu) so that
// the variants compile in parallel.
#pragma once

#include <algorithm>

#include "rq_device.cuh"

namespace clq {

// Per-type launchers (rotate_quant_f16.cu / rotate_quant_bf16.cu); `threads`,
// `smem` and a.rows_per_tile come from rotate_quant_config.
cudaError_t launch_rotate_quant_f16(const RotateQuantArgs& a, int logb, int threads, size_t smem,
                                    int sms, cudaStream_t st);
cudaError_t launch_rotate_quant_bf16(const RotateQuantArgs& a, int logb, int threads,
                                     size_t smem, int sms, cudaStream_t st);

namespace rq {

template <typename T, int LOGB, bool CLIP, int STRIDE, int STAGES, bool SPLIT, bool ASYM>
__global__ void __maxnreg__(kMaxRegs) rotate_quant_kernel(RotateQuantArgs a) {
  extern __shared__ __align__(16) uint8_t smem[];
  run<T, LOGB, CLIP, STRIDE, STAGES, SPLIT, ASYM>(a, smem, nullptr, NoPublish());
}

template <typename T, int LOGB, bool CLIP, int STRIDE, int STAGES, bool SPLIT, bool ASYM>
cudaError_t launch_geom(const RotateQuantArgs& a, int threads, size_t smem, int sms,
                        cudaStream_t st) {
  auto kern = rotate_quant_kernel<T, LOGB, CLIP, STRIDE, STAGES, SPLIT, ASYM>;
  int per_sm = 0;
  cudaError_t e = kernel_setup(reinterpret_cast<const void*>(kern), smem, threads, &per_sm);
  if (e != cudaSuccess) return e;
  if (per_sm < 1) return cudaErrorInvalidConfiguration;
  const int ntiles = (a.M + a.rows_per_tile - 1) / a.rows_per_tile;
  const int g = std::min(ntiles, sms * per_sm);
  return launch_pdl(kern, g, threads, smem, st, a);
}

template <typename T, int LOGB, bool CLIP, bool SPLIT = false, bool ASYM = false>
cudaError_t launch_b(const RotateQuantArgs& a, int threads, size_t smem, int sms,
                     cudaStream_t st) {
  return launch_geom<T, LOGB, CLIP, kStride, kStages, SPLIT, ASYM>(a, threads, smem, sms, st);
}

// log2(b) is a compile-time constant for b >= 16 on the 4-bit activation
// path; smaller blocks, the clipped (weight) path and 8-bit codes read it at
// run time, and so do the asymmetric (a.lo != null) variants.
template <typename T>
cudaError_t launch_rotate_quant_t(const RotateQuantArgs& a, int logb, int threads, size_t smem,
                                  int sms, cudaStream_t st) {
  if (a.lo != nullptr)
    return a.e4m3 == 2 ? launch_b<T, -1, false, true, true>(a, threads, smem, sms, st)
                       : launch_b<T, -1, false, false, true>(a, threads, smem, sms, st);
  if (a.e4m3 == 2)
    return a.clip != nullptr ? launch_b<T, -1, true, true>(a, threads, smem, sms, st)
                             : launch_b<T, -1, false, true>(a, threads, smem, sms, st);
  if (a.clip != nullptr) return launch_b<T, -1, true>(a, threads, smem, sms, st);
  switch (logb) {
    case 4: return launch_b<T, 4, false>(a, threads, smem, sms, st);
    case 5: return launch_b<T, 5, false>(a, threads, smem, sms, st);
    case 6: return launch_b<T, 6, false>(a, threads, smem, sms, st);
    case 7: return launch_b<T, 7, false>(a, threads, smem, sms, st);
    case 8: return launch_b<T, 8, false>(a, threads, smem, sms, st);
    default: return launch_b<T, -1, false>(a, threads, smem, sms, st);
  }
}

}  // namespace rq
}  // namespace clq
