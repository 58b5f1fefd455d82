// Standalone rotate-quantize kernel and its launch templates, instantiated
// once per input type (rotate_quant_f16.cu, rotate_quant_bf16.cu) so that
// the variants compile in parallel.
#pragma once

#include <algorithm>

#include "rq_device.cuh"
#include "rq_pair.cuh"
#include "rq_wide.cuh"

namespace clq {

// Per-type launchers (rotate_quant_f16.cu / rotate_quant_bf16.cu); `threads`,
// `smem` and a.rows_per_tile come from rotate_quant_config.
cudaError_t launch_rotate_quant_f16(const RotateQuantArgs& a, int logb, int threads, size_t smem,
                                    int sms, cudaStream_t st);
cudaError_t launch_rotate_quant_bf16(const RotateQuantArgs& a, int logb, int threads,
                                     size_t smem, int sms, cudaStream_t st);
// Wide-segment kernel per input type and code layout (rotate_quant_pair_*.cu).
cudaError_t launch_rotate_quant_wide_f16_e4m3(const RotateQuantArgs& a, int logb, int stage,
                                              int threads, size_t smem, int sms, cudaStream_t st);
cudaError_t launch_rotate_quant_wide_f16_e2m3(const RotateQuantArgs& a, int logb, int stage,
                                              int threads, size_t smem, int sms, cudaStream_t st);
cudaError_t launch_rotate_quant_wide_bf16_e4m3(const RotateQuantArgs& a, int logb, int stage,
                                               int threads, size_t smem, int sms, cudaStream_t st);
cudaError_t launch_rotate_quant_wide_bf16_e2m3(const RotateQuantArgs& a, int logb, int stage,
                                               int threads, size_t smem, int sms, cudaStream_t st);
// Paired-row kernel per input type and code layout (rotate_quant_pair_*.cu).
cudaError_t launch_rotate_quant_pair_f16_e4m3(const RotateQuantArgs& a, int logb, int half,
                                              int threads, size_t smem, int sms, cudaStream_t st);
cudaError_t launch_rotate_quant_pair_f16_e2m3(const RotateQuantArgs& a, int logb, int half,
                                              int threads, size_t smem, int sms, cudaStream_t st);
cudaError_t launch_rotate_quant_pair_bf16_e4m3(const RotateQuantArgs& a, int logb, int half,
                                               int threads, size_t smem, int sms, cudaStream_t st);
cudaError_t launch_rotate_quant_pair_bf16_e2m3(const RotateQuantArgs& a, int logb, int half,
                                               int threads, size_t smem, int sms, cudaStream_t st);

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
  return launch_ex(kern, g, threads, smem, st, a.serial == 0, a);
}

template <typename T, int LOGB, bool CLIP, bool SPLIT = false, bool ASYM = false>
cudaError_t launch_b(const RotateQuantArgs& a, int threads, size_t smem, int sms,
                     cudaStream_t st) {
  return launch_geom<T, LOGB, CLIP, kStride, kStages, SPLIT, ASYM>(a, threads, smem, sms, st);
}

// Paired-row kernel (rq_pair.cuh): a.rows_per_tile = rows of one half.
template <typename T, int LOGB, int CODES, int HALF, bool ROT>
cudaError_t launch_pair_geom(const RotateQuantArgs& a, int threads, size_t smem, int sms,
                             cudaStream_t st) {
  auto kern = rotate_quant_pair_kernel<T, LOGB, CODES, HALF, kPairStages, ROT>;
  int per_sm = 0;
  cudaError_t e = kernel_setup(reinterpret_cast<const void*>(kern), smem, threads, &per_sm);
  if (e != cudaSuccess) return e;
  if (per_sm < 1) return cudaErrorInvalidConfiguration;
  const int tiles = (a.M + 2 * a.rows_per_tile - 1) / (2 * a.rows_per_tile);
  const int g = std::min(tiles, sms * per_sm);
  return launch_ex(kern, g, threads, smem, st, a.serial == 0, a);
}

template <typename T, int CODES, int HALF, bool ROT>
cudaError_t launch_pair_b(const RotateQuantArgs& a, int logb, int threads, size_t smem, int sms,
                          cudaStream_t st) {
  switch (logb) {
    case 5: return launch_pair_geom<T, 5, CODES, HALF, ROT>(a, threads, smem, sms, st);
    case 6: return launch_pair_geom<T, 6, CODES, HALF, ROT>(a, threads, smem, sms, st);
    case 7: return launch_pair_geom<T, 7, CODES, HALF, ROT>(a, threads, smem, sms, st);
    default: return launch_pair_geom<T, 8, CODES, HALF, ROT>(a, threads, smem, sms, st);
  }
}

template <typename T, int CODES, bool ROT>
cudaError_t launch_pair_h(const RotateQuantArgs& a, int logb, int half, int threads, size_t smem,
                          int sms, cudaStream_t st) {
  return half == kPairHalfSmall
             ? launch_pair_b<T, CODES, kPairHalfSmall, ROT>(a, logb, threads, smem, sms, st)
             : launch_pair_b<T, CODES, kPairHalfLarge, ROT>(a, logb, threads, smem, sms, st);
}

// The paired kernel for CODES (1 E4M3, 3 E2M3), 32 <= b <= 256; `half` is the
// half-stage size rotate_quant_pair_config chose.
template <typename T, int CODES>
cudaError_t launch_rotate_quant_pair_t(const RotateQuantArgs& a, int logb, int half, int threads,
                                       size_t smem, int sms, cudaStream_t st) {
  if (a.rot != nullptr)
    return launch_pair_h<T, CODES, true>(a, logb, half, threads, smem, sms, st);
  return launch_pair_h<T, CODES, false>(a, logb, half, threads, smem, sms, st);
}

// Wide-segment kernel (rq_wide.cuh): a.rows_per_tile = rows of a tile.
template <typename T, int LOGB, int CODES, int STAGE, bool ROT, bool ASYM = false>
cudaError_t launch_wide_geom(const RotateQuantArgs& a, int threads, size_t smem, int sms,
                             cudaStream_t st) {
  auto kern = rotate_quant_wide_kernel<T, LOGB, CODES, STAGE, kPairStages, ROT, ASYM>;
  int per_sm = 0;
  cudaError_t e = kernel_setup(reinterpret_cast<const void*>(kern), smem, threads, &per_sm);
  if (e != cudaSuccess) return e;
  if (per_sm < 1) return cudaErrorInvalidConfiguration;
  const int tiles = (a.M + a.rows_per_tile - 1) / a.rows_per_tile;
  const int g = std::min(tiles, sms * per_sm);
  return launch_ex(kern, g, threads, smem, st, a.serial == 0, a);
}

template <typename T, int CODES, int STAGE, bool ROT>
cudaError_t launch_wide_b(const RotateQuantArgs& a, int logb, int threads, size_t smem, int sms,
                          cudaStream_t st) {
  (void)logb;  // b = 64 only
  if constexpr (CODES == 1)
    if (a.lo != nullptr)
      return launch_wide_geom<T, 6, CODES, STAGE, ROT, true>(a, threads, smem, sms, st);
  return launch_wide_geom<T, 6, CODES, STAGE, ROT>(a, threads, smem, sms, st);
}

// The wide kernel for CODES (1 E4M3, 3 E2M3), b = 64, K % 64 == 0; `stage`
// is the stage size rotate_quant_wide_config chose.
template <typename T, int CODES>
cudaError_t launch_rotate_quant_wide_t(const RotateQuantArgs& a, int logb, int stage, int threads,
                                       size_t smem, int sms, cudaStream_t st) {
  if (a.rot != nullptr)
    return stage == kPairHalfSmall
               ? launch_wide_b<T, CODES, kPairHalfSmall, true>(a, logb, threads, smem, sms, st)
               : launch_wide_b<T, CODES, kPairHalfLarge, true>(a, logb, threads, smem, sms, st);
  return stage == kPairHalfSmall
             ? launch_wide_b<T, CODES, kPairHalfSmall, false>(a, logb, threads, smem, sms, st)
             : launch_wide_b<T, CODES, kPairHalfLarge, false>(a, logb, threads, smem, sms, st);
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
