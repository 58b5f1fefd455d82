// Block-wide helpers for the offline kernels (outlier metrics, clip table).
#pragma once

#include "clq_device.cuh"

namespace clq {

// Sorts v[0 .. n) ascending in shared memory with a bitonic network; n a
// power of two, every thread of the block takes part (ends with a barrier).
__device__ __forceinline__ void bitonic_sort_ascending(float* v, int n) {
  for (int k = 2; k <= n; k <<= 1) {
    for (int j = k >> 1; j > 0; j >>= 1) {
      for (int i = threadIdx.x; i < n; i += blockDim.x) {
        const int ixj = i ^ j;
        if (ixj > i) {
          const bool up = (i & k) == 0;
          const float a = v[i], b = v[ixj];
          if ((a > b) == up) {
            v[i] = b;
            v[ixj] = a;
          }
        }
      }
      __syncthreads();
    }
  }
}

}  // namespace clq
