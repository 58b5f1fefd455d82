// Peak-rate microbenchmarks: the measured denominators the measurement
// reports next to the GEMM and rotate-quant rates.  Each launcher only
// launches; the caller times the launch with CUDA events on `stream` and
// divides the operation count the launcher returns by the elapsed time.
//  * tcgen05 E4M3 (kind::f8f6f4, the MMA the GEMM uses): one CTA per SM, one
//    thread issues back-to-back 128 x 256 x 32 MMAs on fixed shared-memory
//    operands into one TMEM accumulator;
//  * mma.sync (warp-level MMA, the only INT8 / INT4 tensor path sm_103a
//    has): s8 m16n8k32, s4 m16n8k64 and, for comparison, e4m3 m16n8k32,
//    8 warps per CTA, 4 CTAs per SM, 4 independent accumulators per warp;
//  * HBM read: every byte of a caller buffer read once with 16-byte loads;
//  * operand stream: the W4A4 GEMM's main loop without its epilogue, one CTA
//    per SM: a TMA producer fills a ring of four 48 KB stages with the GEMM's
//    boxes (A 128 rows, B 256 rows, 128 codes a row, E4M3 or E2M3 layout)
//    from a caller code array, and a consumer either releases each stage at
//    once (the rate at which an SM takes operands in) or issues the GEMM's
//    four 128 x 256 x 32 MMAs on it (the rate of the main loop);
//  * rotate-quant stream: the wide rotate-quant loop's data movement without
//    its arithmetic (its tiles, stage ring, threads and programmatic-launch
//    prologue; one byte out per element and four per row), the memory floor
//    the kernel is measured against.
#include "clq_device.cuh"
#include "clq_kernels.h"

namespace clq {

namespace {

constexpr int kPeakA = 128 * 128;  // bytes: 128 rows x one 128-byte swizzle row
constexpr int kPeakB = 256 * 128;

__global__ void __launch_bounds__(128, 1) peak_tcgen05_kernel(int iters, int32_t* status) {
  extern __shared__ uint8_t smem_raw[];
  __shared__ uint64_t bar;
  __shared__ uint32_t slot;
  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  for (int i = threadIdx.x; i < (kPeakA + kPeakB) / 16; i += blockDim.x)
    reinterpret_cast<uint4*>(smem)[i] = make_uint4(0u, 0u, 0u, 0u);
  fence_proxy_async_smem();
  if (threadIdx.x == 0) {
    mbar_init(&bar, 1);
    fence_mbarrier_init();
  }
  if (threadIdx.x < 32) {
    tmem_alloc(&slot, 256);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = slot;
  if (threadIdx.x == 0) {
    constexpr uint32_t idesc = idesc_e4m3_f32(128, 256);
    const uint32_t a0 = smem_addr(smem), b0 = smem_addr(smem + kPeakA);
#pragma unroll 1
    for (int i = 0; i < iters; ++i) {
#pragma unroll
      for (int k = 0; k < 4; ++k)
        mma_e4m3(tmem, sw128_desc(a0 + 32 * k), sw128_desc(b0 + 32 * k), idesc,
                 (i | k) != 0 ? 1u : 0u);
    }
    mma_commit(&bar);
    mbar_wait_bounded(&bar, 0, nullptr, status, 2000000000ull);
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (threadIdx.x < 32) tmem_dealloc(tmem, 256);
}

template <int KIND>
__device__ __forceinline__ void mma_sync_step(uint32_t (&c)[4], const uint32_t (&a)[4],
                                              const uint32_t (&b)[2]) {
  if (KIND == 0)
    asm volatile(
        "mma.sync.aligned.m16n8k32.row.col.s32.s8.s8.s32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, "
        "{%8,%9}, {%0,%1,%2,%3};"
        : "+r"(c[0]), "+r"(c[1]), "+r"(c[2]), "+r"(c[3])
        : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b[0]), "r"(b[1]));
  else if (KIND == 1)
    asm volatile(
        "mma.sync.aligned.m16n8k64.row.col.s32.s4.s4.s32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, "
        "{%8,%9}, {%0,%1,%2,%3};"
        : "+r"(c[0]), "+r"(c[1]), "+r"(c[2]), "+r"(c[3])
        : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b[0]), "r"(b[1]));
  else
    asm volatile(
        "mma.sync.aligned.m16n8k32.row.col.f32.e4m3.e4m3.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, "
        "{%8,%9}, {%0,%1,%2,%3};"
        : "+r"(c[0]), "+r"(c[1]), "+r"(c[2]), "+r"(c[3])
        : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b[0]), "r"(b[1]));
}

template <int KIND>
__global__ void __launch_bounds__(256) peak_mma_sync_kernel(int iters, int32_t* sink) {
  const uint32_t t = threadIdx.x;
  const uint32_t a[4] = {t * 0x01010101u, t ^ 0x55u, t + 7u, t * 3u};
  const uint32_t b[2] = {t ^ 0x33u, t * 5u};
  uint32_t c[4][4] = {};
#pragma unroll 1
  for (int i = 0; i < iters; ++i) {
#pragma unroll
    for (int j = 0; j < 4; ++j) mma_sync_step<KIND>(c[j], a, b);
  }
  uint32_t x = 0;
#pragma unroll
  for (int j = 0; j < 4; ++j) x ^= c[j][0] ^ c[j][1] ^ c[j][2] ^ c[j][3];
  if (x == 0x9E3779B9u) sink[0] = static_cast<int32_t>(x);  // keeps the loop alive
}

__global__ void peak_hbm_read_kernel(const uint4* __restrict__ p, size_t n, int32_t* sink) {
  uint32_t x = 0;
  for (size_t i = blockIdx.x * static_cast<size_t>(blockDim.x) + threadIdx.x; i < n;
       i += static_cast<size_t>(gridDim.x) * blockDim.x) {
    const uint4 v = __ldcs(p + i);
    x ^= v.x ^ v.y ^ v.z ^ v.w;
  }
  if (x == 0x9E3779B9u) sink[0] = static_cast<int32_t>(x);
}

constexpr int kStreamStages = 4;
constexpr int kStreamA = 128 * 128;  // smem bytes of one A box (E4M3 or padded E2M3)
constexpr int kStreamB = 256 * 128;

// F6: E2M3 boxes (0.75 of the smem bytes cross from L2); MMA: issue the MMAs.
template <bool F6, bool MMA>
__global__ void __launch_bounds__(128, 1)
    peak_stream_kernel(const __grid_constant__ CUtensorMap mapA,
                       const __grid_constant__ CUtensorMap mapB, int rows, int K, int tiles,
                       int32_t* status) {
  extern __shared__ uint8_t smem_raw[];
  __shared__ __align__(8) uint64_t full[kStreamStages], empty[kStreamStages], done;
  __shared__ uint32_t slot;
  __shared__ int32_t abort;
  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    for (int s = 0; s < kStreamStages; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    mbar_init(&done, 1);
    abort = 0;
    fence_mbarrier_init();
  }
  if (MMA && warp == 1) {
    tmem_alloc(&slot, 256);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const int nk = K / 128, mt = rows / 128, nt = rows / 256;
  constexpr uint32_t TX = F6 ? (kStreamA + kStreamB) / 4 * 3 : kStreamA + kStreamB;
  const int steps = tiles * nk;
  if (warp == 0 && lane == 0) {
    prefetch_tensor_map(&mapA);
    prefetch_tensor_map(&mapB);
    for (int it = 0; it < steps; ++it) {
      const int s = it % kStreamStages;
      const int t = static_cast<int>(blockIdx.x) + (it / nk) * static_cast<int>(gridDim.x);
      const int kb = it % nk;
      if (!mbar_wait_bounded(&empty[s], ((it / kStreamStages) & 1) ^ 1, &abort, status,
                             kWaitLimitNs))
        break;
      mbar_arrive_expect_tx(&full[s], TX);
      uint8_t* st = smem + s * (kStreamA + kStreamB);
      tma_load_2d(st, &mapA, kb * 128, (t % mt) * 128, &full[s]);
      tma_load_2d(st + kStreamA, &mapB, kb * 128, ((t / mt) % nt) * 256, &full[s]);
    }
  } else if (warp == 1 && lane == 0) {
    constexpr uint32_t idesc = F6 ? idesc_f8f6f4_f32(128, 256, kFmtE2M3, kFmtE2M3)
                                  : idesc_e4m3_f32(128, 256);
    bool ok = true;
    for (int it = 0; it < steps && ok; ++it) {
      const int s = it % kStreamStages;
      ok = mbar_wait_bounded(&full[s], (it / kStreamStages) & 1, &abort, status, kWaitLimitNs);
      if (!ok) break;
      if (MMA) {
        tc_fence_after();
        const uint32_t a0 = smem_addr(smem + s * (kStreamA + kStreamB));
        const uint32_t b0 = a0 + kStreamA;
#pragma unroll
        for (int k = 0; k < 4; ++k)
          mma_e4m3(slot, sw128_desc(a0 + 32 * k), sw128_desc(b0 + 32 * k), idesc,
                   (it | k) != 0 ? 1u : 0u);
        mma_commit(&empty[s]);
      } else {
        mbar_arrive(&empty[s]);
      }
    }
    if (MMA) {
      mma_commit(&done);
      mbar_wait_bounded(&done, 0, nullptr, nullptr, 100000000ull);
    }
    if (!ok) {  // copies already issued land before the CTA exits
      for (int s = 0; s < kStreamStages; ++s)
        for (int ph = 0; ph < 2; ++ph)
          mbar_wait_bounded(&full[s], ph, nullptr, nullptr, 10000000ull);
    }
  }
  tc_fence_before();
  __syncthreads();
  if (MMA && warp == 1) {
    tc_fence_after();
    tmem_dealloc(slot, 256);
  }
}

template <bool F6, bool MMA>
cudaError_t launch_stream_t(const CUtensorMap& a, const CUtensorMap& b, int rows, int K,
                            int tiles, int32_t* status, int sms, cudaStream_t st) {
  auto k = peak_stream_kernel<F6, MMA>;
  const size_t smem = kStreamStages * (kStreamA + kStreamB) + 1024;
  cudaError_t e = kernel_setup(reinterpret_cast<const void*>(k), smem, 128, nullptr);
  if (e != cudaSuccess) return e;
  k<<<sms, 128, smem, st>>>(a, b, rows, K, tiles, status);
  return cudaGetLastError();
}

// Rotate-quant memory floor.  Tiles of RH rows of 2K bytes are dealt
// round-robin and bulk-copied into a ring of two STAGE-byte stages (the
// first two into L2 before the programmatic-launch wait), as in the wide
// rotate-quant loop; each thread then turns its 16-element chunks of a tile
// into 16 bytes (the high byte of every 16-bit value) and the first RH
// threads write a 4-byte value per row: the loop's HBM traffic (2 B in,
// 1 B + 4 B a row out) with no gather and no arithmetic.
template <int STAGE>
__global__ void __launch_bounds__(512) peak_rq_stream_kernel(const uint8_t* X, int M, int K,
                                                             int RH, uint8_t* Q, float* S,
                                                             int32_t* status) {
  extern __shared__ __align__(16) uint8_t smem[];
  __shared__ __align__(8) uint64_t full[2];
  const int tid = threadIdx.x;
  const int ntiles = (M + RH - 1) / RH;
  const uint32_t row_bytes = 2u * static_cast<uint32_t>(K);
  auto rows_of = [&](int t) { return min(RH, M - t * RH); };
  auto src_of = [&](int t) { return X + static_cast<size_t>(t) * RH * row_bytes; };
  if (tid == 0) {
    mbar_init(&full[0], 1);
    mbar_init(&full[1], 1);
    fence_mbarrier_init();
  }
  __syncthreads();
  if (tid == 0)
    for (int s = 0; s < 2; ++s) {
      const int t = static_cast<int>(blockIdx.x) + s * static_cast<int>(gridDim.x);
      if (t < ntiles) bulk_prefetch_l2(src_of(t), row_bytes * static_cast<uint32_t>(rows_of(t)));
    }
  pdl_wait();
  pdl_launch_dependents();
  auto issue = [&](int s, int t) {
    const uint32_t bytes = row_bytes * static_cast<uint32_t>(rows_of(t));
    mbar_arrive_expect_tx(&full[s], bytes);
    bulk_load(smem + s * STAGE, src_of(t), bytes, &full[s]);
  };
  if (tid == 0)
    for (int s = 0; s < 2; ++s) {
      const int t = static_cast<int>(blockIdx.x) + s * static_cast<int>(gridDim.x);
      if (t < ntiles) issue(s, t);
    }
  for (int j = 0;; ++j) {
    const int s = j & 1;
    const int t = static_cast<int>(blockIdx.x) + j * static_cast<int>(gridDim.x);
    if (t >= ntiles) break;
    if (!mbar_wait_bounded(&full[s], (j >> 1) & 1, nullptr, status, kWaitLimitNs)) {
      if (tid == 0)  // copies already issued land before the CTA exits
        for (int s2 = 0; s2 < 2; ++s2)
          for (int ph = 0; ph < 2; ++ph)
            mbar_wait_bounded(&full[s2], ph, nullptr, nullptr, 10000000ull);
      break;
    }
    const int rows = rows_of(t);
    const int n16 = rows * K / 16;
    const uint8_t* stage = smem + s * STAGE;
    uint4* q = reinterpret_cast<uint4*>(Q + static_cast<size_t>(t) * RH * K);
    for (int i = tid; i < n16; i += blockDim.x) {
      const uint4 a = *reinterpret_cast<const uint4*>(stage + 32 * i);
      const uint4 b = *reinterpret_cast<const uint4*>(stage + 32 * i + 16);
      q[i] = make_uint4(__byte_perm(a.x, a.y, 0x7531), __byte_perm(a.z, a.w, 0x7531),
                        __byte_perm(b.x, b.y, 0x7531), __byte_perm(b.z, b.w, 0x7531));
    }
    if (tid < rows) S[t * RH + tid] = 1.0f;
    __syncthreads();  // stage s fully read
    if (tid == 0) {
      const int t2 = t + 2 * static_cast<int>(gridDim.x);
      if (t2 < ntiles) issue(s, t2);
    }
  }
}

template <int STAGE>
cudaError_t launch_rq_stream_t(const uint8_t* X, int M, int K, int RH, int threads, uint8_t* Q,
                               float* S, int32_t* status, int sms, cudaStream_t st) {
  auto k = peak_rq_stream_kernel<STAGE>;
  const size_t smem = 2 * STAGE;
  int per_sm = 0;
  cudaError_t e = kernel_setup(reinterpret_cast<const void*>(k), smem, threads, &per_sm);
  if (e != cudaSuccess) return e;
  if (per_sm < 1) return cudaErrorInvalidConfiguration;
  const int tiles = (M + RH - 1) / RH;
  return launch_pdl(k, std::min(tiles, sms * per_sm), threads, smem, st, X, M, K, RH, Q, S,
                    status);
}

}  // namespace

// The wide loop's geometry (rotate_quant.cu).
void rotate_quant_wide_config(int M, int K, int sms, int* rows, int* threads, size_t* smem,
                              int* stage);

cudaError_t launch_peak_rq_stream(const void* X, int M, int K, uint8_t* Q, float* S,
                                  int32_t* status, cudaStream_t st, long long* bytes) {
  const int sms = sm_count();
  if (sms <= 0) return cudaErrorInvalidDevice;
  int RH = 0, threads = 0, stage = 0;
  size_t smem = 0;
  rotate_quant_wide_config(M, K, sms, &RH, &threads, &smem, &stage);
  *bytes = static_cast<long long>(M) * (5LL * K / 2 + 4);
  const uint8_t* x = static_cast<const uint8_t*>(X);
  if (stage == 16 * 1024)
    return launch_rq_stream_t<16384>(x, M, K, RH, threads, Q, S, status, sms, st);
  return launch_rq_stream_t<32768>(x, M, K, RH, threads, Q, S, status, sms, st);
}

cudaError_t launch_peak_operand_stream(const uint8_t* buf, int rows, int K, int codes, int mma,
                                       int tiles, int32_t* status, cudaStream_t st,
                                       long long* smem_bytes, long long* macs) {
  const int sms = sm_count();
  if (sms <= 0) return cudaErrorInvalidDevice;
  CUtensorMap a, b;
  if (!encode_codes_map(&a, buf, codes, rows, K, 128, 0) ||
      !encode_codes_map(&b, buf, codes, rows, K, 256, 0))
    return cudaErrorInvalidValue;
  const long long steps = static_cast<long long>(sms) * tiles * (K / 128);
  *smem_bytes = steps * (kStreamA + kStreamB);
  *macs = mma ? steps * 128LL * 256 * 128 : 0;

  const bool f6 = codes == CLQ_CODES_E2M3;
  if (f6)
    return mma ? launch_stream_t<true, true>(a, b, rows, K, tiles, status, sms, st)
               : launch_stream_t<true, false>(a, b, rows, K, tiles, status, sms, st);
  return mma ? launch_stream_t<false, true>(a, b, rows, K, tiles, status, sms, st)
             : launch_stream_t<false, false>(a, b, rows, K, tiles, status, sms, st);
}

cudaError_t launch_peak_tcgen05(int iters, int32_t* status, cudaStream_t st, long long* macs) {
  const int sms = sm_count();
  if (sms <= 0) return cudaErrorInvalidDevice;
  const size_t smem = kPeakA + kPeakB + 1024;
  cudaError_t e = kernel_setup(reinterpret_cast<const void*>(peak_tcgen05_kernel), smem, 128,
                               nullptr);
  if (e != cudaSuccess) return e;
  peak_tcgen05_kernel<<<sms, 128, smem, st>>>(iters, status);
  *macs = static_cast<long long>(sms) * iters * 4 * 128 * 256 * 32;
  return cudaGetLastError();
}

cudaError_t launch_peak_mma_sync(int kind, int iters, int32_t* sink, cudaStream_t st,
                                 long long* macs) {
  const int sms = sm_count();
  if (sms <= 0) return cudaErrorInvalidDevice;
  const int grid = 4 * sms, threads = 256;
  const long long per = kind == 1 ? 16 * 8 * 64 : 16 * 8 * 32;  // MACs per warp MMA
  *macs = static_cast<long long>(grid) * (threads / 32) * iters * 4 * per;
  if (kind == 0)
    peak_mma_sync_kernel<0><<<grid, threads, 0, st>>>(iters, sink);
  else if (kind == 1)
    peak_mma_sync_kernel<1><<<grid, threads, 0, st>>>(iters, sink);
  else
    peak_mma_sync_kernel<2><<<grid, threads, 0, st>>>(iters, sink);
  return cudaGetLastError();
}

cudaError_t launch_peak_hbm_read(const void* buf, size_t bytes, int32_t* sink, cudaStream_t st) {
  const int sms = sm_count();
  if (sms <= 0) return cudaErrorInvalidDevice;
  peak_hbm_read_kernel<<<8 * sms, 512, 0, st>>>(static_cast<const uint4*>(buf), bytes / 16,
                                                sink);
  return cudaGetLastError();
}

}  // namespace clq
