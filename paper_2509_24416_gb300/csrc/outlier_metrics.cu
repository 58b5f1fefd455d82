// Outlier scores under the alternative metrics of arxiv 2509.24416 Sec. 4.4
// ("Choice of Outlier Metric": percentile (1 %, 99 %), top-k mean with
// k = 1 %, range, peak-to-average ratio), next to Sec. 3.3's absolute
// maximum.  Offline, once per layer.  The scores decide an integer
// permutation, so every step is taken in fp32 in one fixed order, the one
// the CPU oracle takes:
//   S[t] = (sum over b in order of calib[b][t][c]) / B;
//   absmax     max_t |S|;
//   range      max_t S - min_t S;
//   par        max_t |S| / ((sum over t in order of |S|) / T), 0 if the sum is 0;
//   percentile max(|P(0.01)|, |P(0.99)|), P(q) = v[lo] + (pos - lo)(v[lo+1] - v[lo])
//              over the ascending order statistics v, pos = q (T - 1), lo = floor(pos);
//   topk_mean  (sum of the k largest |S|, largest first) / k, k = max(1, (T + 50) / 100).
// One CTA per channel holds S (T <= 16384 values) in shared memory and sorts
// it with a bitonic network where an order statistic is needed.
#include "clq_device.cuh"
#include "clq_kernels.h"
#include "sort_util.cuh"

namespace clq {

namespace {

constexpr int kThreads = 256;

// Block-wide max of x (every thread contributes); the result in every thread.
__device__ __forceinline__ float block_max(float x, float* red) {
  for (int o = 16; o > 0; o >>= 1) x = fmaxf(x, __shfl_xor_sync(0xffffffffu, x, o));
  const int w = threadIdx.x >> 5;
  if ((threadIdx.x & 31) == 0) red[w] = x;
  __syncthreads();
  float r = red[0];
  for (int i = 1; i < kThreads / 32; ++i) r = fmaxf(r, red[i]);
  __syncthreads();
  return r;
}

__device__ __forceinline__ float percentile_fp32(const float* v, int n, float q) {
  const float pos = __fmul_rn(q, static_cast<float>(n - 1));
  const int lo = static_cast<int>(floorf(pos));
  const int hi = min(lo + 1, n - 1);
  const float frac = __fsub_rn(pos, static_cast<float>(lo));
  return __fadd_rn(v[lo], __fmul_rn(frac, __fsub_rn(v[hi], v[lo])));
}

template <typename T>
__global__ void __launch_bounds__(kThreads) outlier_metric_kernel(const uint16_t* calib, int B,
                                                                  int Tn, int K, int Tp,
                                                                  int metric, float* scores) {
  extern __shared__ float v[];  // [Tp]
  __shared__ float red[kThreads / 32];
  const int c = blockIdx.x;
  const size_t bstride = static_cast<size_t>(Tn) * K;
  const float fb = static_cast<float>(B);
  // S[t], and what the metric sorts: S (percentile), -|S| (top-k: ascending
  // order puts the largest magnitudes first).  Padding sorts to the end.
  float lmax = 0.f, lmin = 0.f, labs = 0.f;
  bool any = false;
  for (int t = threadIdx.x; t < Tp; t += blockDim.x) {
    float x = 0.f;
    if (t < Tn) {
      float s = 0.f;
      for (int b = 0; b < B; ++b)
        s = __fadd_rn(s, Num<T>::to_f(calib[b * bstride + static_cast<size_t>(t) * K + c]));
      x = __fdiv_rn(s, fb);
      lmax = any ? fmaxf(lmax, x) : x;
      lmin = any ? fminf(lmin, x) : x;
      labs = fmaxf(labs, fabsf(x));
      any = true;
    }
    if (metric == CLQ_METRIC_TOPK_MEAN)
      v[t] = t < Tn ? -fabsf(x) : __int_as_float(0x7f800000);  // +inf pad
    else
      v[t] = t < Tn ? x : __int_as_float(0x7f800000);
  }
  __syncthreads();
  // Block extremes (threads without a token hold neutral values).
  const float mx = block_max(any ? lmax : -__int_as_float(0x7f800000), red);
  const float mn = -block_max(any ? -lmin : -__int_as_float(0x7f800000), red);
  const float peak = block_max(labs, red);
  if (metric == CLQ_METRIC_PERCENTILE || metric == CLQ_METRIC_TOPK_MEAN)
    bitonic_sort_ascending(v, Tp);
  if (threadIdx.x != 0) return;
  float out = 0.f;
  switch (metric) {
    case CLQ_METRIC_ABSMAX:
      out = peak;
      break;
    case CLQ_METRIC_RANGE:
      out = __fsub_rn(mx, mn);
      break;
    case CLQ_METRIC_PAR: {
      float sum = 0.f;
      for (int t = 0; t < Tn; ++t) sum = __fadd_rn(sum, fabsf(v[t]));
      const float mean = __fdiv_rn(sum, static_cast<float>(Tn));
      out = mean > 0.f ? __fdiv_rn(peak, mean) : 0.f;
      break;
    }
    case CLQ_METRIC_PERCENTILE: {
      const float lo = percentile_fp32(v, Tn, 0.01f);
      const float hi = percentile_fp32(v, Tn, 0.99f);
      out = fmaxf(fabsf(lo), fabsf(hi));
      break;
    }
    default: {  // CLQ_METRIC_TOPK_MEAN
      const int k = max(1, (Tn + 50) / 100);
      float sum = 0.f;
      for (int i = 0; i < k; ++i) sum = __fadd_rn(sum, -v[i]);
      out = __fdiv_rn(sum, static_cast<float>(k));
      break;
    }
  }
  scores[c] = out;
}

}  // namespace

cudaError_t launch_outlier_metric(const void* calib, int dtype, int B, int T, int K, int metric,
                                  float* scores, cudaStream_t st) {
  int Tp = 1;
  while (Tp < T) Tp <<= 1;
  const size_t smem = static_cast<size_t>(Tp) * sizeof(float);
  const uint16_t* c = static_cast<const uint16_t*>(calib);
  if (dtype == CLQ_F16) {
    auto k = outlier_metric_kernel<__half>;
    cudaError_t e = kernel_setup(reinterpret_cast<const void*>(k), smem, kThreads, nullptr);
    if (e != cudaSuccess) return e;
    k<<<K, kThreads, smem, st>>>(c, B, T, K, Tp, metric, scores);
  } else {
    auto k = outlier_metric_kernel<__nv_bfloat16>;
    cudaError_t e = kernel_setup(reinterpret_cast<const void*>(k), smem, kThreads, nullptr);
    if (e != cudaSuccess) return e;
    k<<<K, kThreads, smem, st>>>(c, B, T, K, Tp, metric, scores);
  }
  return cudaGetLastError();
}

}  // namespace clq
