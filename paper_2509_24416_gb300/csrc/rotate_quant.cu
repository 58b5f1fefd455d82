// Standalone rotate-quantize kernel (activations online, weights offline)
// and the outlier-score kernel.  The tile loop itself lives in rq_device.cuh.
#include "rq_device.cuh"

namespace clq {

namespace {

constexpr int kStages = rq::kMaxStages;  // raw tiles in flight per CTA

template <typename T, int LOGB, bool CLIP>
__global__ void __maxnreg__(96) rotate_quant_kernel(RotateQuantArgs a) {
  extern __shared__ __align__(16) uint8_t smem[];
  rq::run<T, LOGB, CLIP>(a, smem, kStages, nullptr, rq::NoPublish());
}

// Outlier score (Sec. 3.3): S = fp32 batch mean (sequential sum over the
// batch, then / B), score[k] = max_t |S[t][k]|.  Threads own channels;
// blockIdx.y owns a slice of tokens; slices combine with an integer atomicMax
// on the (non-negative) float bits, so `scores` must be zeroed first.
template <typename T>
__global__ void outlier_scores_kernel(const uint16_t* calib, int B, int Tn, int K,
                                      int tokens_per_slice, float* scores) {
  const int k = blockIdx.x * blockDim.x + threadIdx.x;
  if (k >= K) return;
  const int t0 = blockIdx.y * tokens_per_slice;
  const int t1 = min(Tn, t0 + tokens_per_slice);
  const size_t bstride = static_cast<size_t>(Tn) * K;
  const float fb = static_cast<float>(B);
  float best = 0.f;
  for (int t = t0; t < t1; ++t) {
    float sum = 0.f;
    for (int b = 0; b < B; ++b)
      sum = sum + Num<T>::to_f(calib[b * bstride + static_cast<size_t>(t) * K + k]);
    best = fmaxf(best, fabsf(__fdiv_rn(sum, fb)));
  }
  atomicMax(reinterpret_cast<unsigned*>(scores) + k, __float_as_uint(best));
}

template <typename T, int LOGB, bool CLIP>
cudaError_t launch_rq_t(const RotateQuantArgs& a, int threads, size_t smem, int sms,
                        cudaStream_t st) {
  auto kern = rotate_quant_kernel<T, LOGB, CLIP>;
  int per_sm = 0;
  cudaError_t e = kernel_setup(reinterpret_cast<const void*>(kern), smem, threads, &per_sm);
  if (e != cudaSuccess) return e;
  if (per_sm < 1) return cudaErrorInvalidConfiguration;
  const int ntiles = (a.M + a.rows_per_tile - 1) / a.rows_per_tile;
  const int g = std::min(ntiles, sms * per_sm);
  kern<<<g, threads, smem, st>>>(a);
  return cudaGetLastError();
}

template <typename T, bool CLIP>
cudaError_t launch_rq_b(const RotateQuantArgs& a, int logb, int threads, size_t smem, int sms,
                        cudaStream_t st) {
  switch (logb) {
    case 0: return launch_rq_t<T, 0, CLIP>(a, threads, smem, sms, st);
    case 1: return launch_rq_t<T, 1, CLIP>(a, threads, smem, sms, st);
    case 2: return launch_rq_t<T, 2, CLIP>(a, threads, smem, sms, st);
    case 3: return launch_rq_t<T, 3, CLIP>(a, threads, smem, sms, st);
    case 4: return launch_rq_t<T, 4, CLIP>(a, threads, smem, sms, st);
    case 5: return launch_rq_t<T, 5, CLIP>(a, threads, smem, sms, st);
    case 6: return launch_rq_t<T, 6, CLIP>(a, threads, smem, sms, st);
    case 7: return launch_rq_t<T, 7, CLIP>(a, threads, smem, sms, st);
    case 8: return launch_rq_t<T, 8, CLIP>(a, threads, smem, sms, st);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace

// Rows per tile: the CTA gets one thread per 32-element segment of each of
// its rows.  Prefer thread counts that fill whole warps (padding lanes do no
// useful work) and lie in [192, 384], which keeps two CTAs per SM, and keep
// the shared-memory footprint (S + 1 row buffers) under 113 KB.
void rotate_quant_config(int K, int* rows_per_tile, int* threads, size_t* smem) {
  const int segs = K >> 5;
  int best_r = 1;
  double best_score = -1.0;
  for (int r = 1; r * segs <= 512; ++r) {
    if (r > 1 && rq::smem_bytes(K, r, kStages) > 113u * 1024u) break;
    const int t = r * segs;
    const int t32 = (t + 31) & ~31;
    const double fill = static_cast<double>(t) / t32;
    const double size_term =
        t32 < 192 ? t32 / 384.0 : (t32 <= 384 ? 1.0 + t32 / 4096.0 : 0.5);
    const double score = fill * 4.0 + size_term;
    if (score > best_score + 1e-9) {
      best_score = score;
      best_r = r;
    }
  }
  *rows_per_tile = best_r;
  *threads = ((best_r * segs) + 31) & ~31;
  *smem = rq::smem_bytes(K, best_r, kStages);
}

cudaError_t launch_rotate_quant(const RotateQuantArgs& a, int dtype, int logb,
                                cudaStream_t st) {
  RotateQuantArgs args = a;
  int threads = 0;
  size_t smem = 0;
  rotate_quant_config(a.K, &args.rows_per_tile, &threads, &smem);
  const int sms = sm_count();
  if (sms <= 0) return cudaErrorInvalidDevice;
  const bool clip = a.clip != nullptr;
  if (dtype == CLQ_F16)
    return clip ? launch_rq_b<__half, true>(args, logb, threads, smem, sms, st)
                : launch_rq_b<__half, false>(args, logb, threads, smem, sms, st);
  return clip ? launch_rq_b<__nv_bfloat16, true>(args, logb, threads, smem, sms, st)
              : launch_rq_b<__nv_bfloat16, false>(args, logb, threads, smem, sms, st);
}

cudaError_t launch_outlier_scores(const void* calib, int dtype, int B, int T, int K,
                                  float* scores, cudaStream_t st) {
  cudaError_t e = cudaMemsetAsync(scores, 0, sizeof(float) * static_cast<size_t>(K), st);
  if (e != cudaSuccess) return e;
  const int threads = 256;
  const int gx = (K + threads - 1) / threads;
  const int slices = std::max(1, std::min(T, 4096 / std::max(gx, 1)));
  const int per = (T + slices - 1) / slices;
  const dim3 grid(gx, (T + per - 1) / per);
  const uint16_t* c = static_cast<const uint16_t*>(calib);
  if (dtype == CLQ_F16)
    outlier_scores_kernel<__half><<<grid, threads, 0, st>>>(c, B, T, K, per, scores);
  else
    outlier_scores_kernel<__nv_bfloat16><<<grid, threads, 0, st>>>(c, B, T, K, per, scores);
  return cudaGetLastError();
}

}  // namespace clq
