// Kernels of the per-layer clip search (arxiv 2509.24416 Sec. 3.4, Eq. 3,
// with the layer as its own target): the table of the J largest |W~[n][k]|
// of every rotated weight row, the gather of one clip vector from it, and a
// deterministic sum of squared output errors.  Offline; the product inside
// the search is the library's own rotate-quant + GEMM.
#include "clq_device.cuh"
#include "clq_kernels.h"
#include "sort_util.cuh"

namespace clq {

namespace {

constexpr int kThreads = 256;

// table[n][j] = j-th largest |w_rot[n][k]| (j < J), one CTA per row: -|w| is
// sorted ascending in shared memory (+inf padding sorts last).
__global__ void __launch_bounds__(kThreads) clip_table_kernel(const float* __restrict__ w_rot,
                                                              int K, int Kp, int J,
                                                              float* __restrict__ table) {
  extern __shared__ float v[];  // [Kp]
  const int n = blockIdx.x;
  const float* row = w_rot + static_cast<size_t>(n) * K;
  for (int k = threadIdx.x; k < Kp; k += blockDim.x)
    v[k] = k < K ? -fabsf(row[k]) : __int_as_float(0x7f800000);
  __syncthreads();
  bitonic_sort_ascending(v, Kp);
  for (int j = threadIdx.x; j < J; j += blockDim.x)
    table[static_cast<size_t>(n) * J + j] = -v[j];
}

__global__ void clip_gather_kernel(const float* __restrict__ table, int N, int J, int j,
                                   float* __restrict__ clip) {
  const int n = blockIdx.x * blockDim.x + threadIdx.x;
  if (n < N) clip[n] = table[static_cast<size_t>(n) * J + j];
}

// partial[blockIdx.x] = sum over this block's grid-stride share of
// (yh - yref)^2 in fp64; the block's sum is a fixed-order tree.
template <typename T>
__global__ void __launch_bounds__(kThreads) sq_err_partial_kernel(const uint16_t* __restrict__ yh,
                                                                  const float* __restrict__ yref,
                                                                  size_t n,
                                                                  double* __restrict__ partial) {
  __shared__ double red[kThreads];
  double acc = 0.0;
  for (size_t i = blockIdx.x * static_cast<size_t>(kThreads) + threadIdx.x; i < n;
       i += static_cast<size_t>(gridDim.x) * kThreads) {
    const double d = static_cast<double>(Num<T>::to_f(yh[i])) - static_cast<double>(yref[i]);
    acc = fma(d, d, acc);
  }
  red[threadIdx.x] = acc;
  __syncthreads();
  for (int s = kThreads / 2; s > 0; s >>= 1) {
    if (threadIdx.x < s) red[threadIdx.x] += red[threadIdx.x + s];
    __syncthreads();
  }
  if (threadIdx.x == 0) partial[blockIdx.x] = red[0];
}

// out[g] = sum_b partial[g][b] in a fixed order, one CTA per grid point.
__global__ void __launch_bounds__(kThreads) sum_partials_kernel(const double* __restrict__ partial,
                                                                int P, double* __restrict__ out) {
  __shared__ double red[kThreads];
  double acc = 0.0;
  for (int b = threadIdx.x; b < P; b += kThreads)
    acc += partial[static_cast<size_t>(blockIdx.x) * P + b];
  red[threadIdx.x] = acc;
  __syncthreads();
  for (int s = kThreads / 2; s > 0; s >>= 1) {
    if (threadIdx.x < s) red[threadIdx.x] += red[threadIdx.x + s];
    __syncthreads();
  }
  if (threadIdx.x == 0) out[blockIdx.x] = red[0];
}

}  // namespace

cudaError_t launch_clip_table(const float* w_rot, int N, int K, int J, float* table,
                              cudaStream_t st) {
  int Kp = 1;
  while (Kp < K) Kp <<= 1;
  const size_t smem = static_cast<size_t>(Kp) * sizeof(float);
  cudaError_t e = kernel_setup(reinterpret_cast<const void*>(clip_table_kernel), smem, kThreads,
                               nullptr);
  if (e != cudaSuccess) return e;
  clip_table_kernel<<<N, kThreads, smem, st>>>(w_rot, K, Kp, J, table);
  return cudaGetLastError();
}

cudaError_t launch_clip_gather(const float* table, int N, int J, int j, float* clip,
                               cudaStream_t st) {
  clip_gather_kernel<<<(N + 255) / 256, 256, 0, st>>>(table, N, J, j, clip);
  return cudaGetLastError();
}

cudaError_t launch_sq_err_partial(const void* yh, int dtype, const float* yref, size_t n,
                                  double* partial, int P, cudaStream_t st) {
  const uint16_t* y = static_cast<const uint16_t*>(yh);
  if (dtype == CLQ_F16)
    sq_err_partial_kernel<__half><<<P, kThreads, 0, st>>>(y, yref, n, partial);
  else
    sq_err_partial_kernel<__nv_bfloat16><<<P, kThreads, 0, st>>>(y, yref, n, partial);
  return cudaGetLastError();
}

cudaError_t launch_sum_partials(const double* partial, int G, int P, double* out,
                                cudaStream_t st) {
  sum_partials_kernel<<<G, kThreads, 0, st>>>(partial, P, out);
  return cudaGetLastError();
}

}  // namespace clq
