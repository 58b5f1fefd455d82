// Packed INT4 x INT4 GEMM with the dequant + bias epilogue on tcgen05.
//
// acc[i][n] = sum_k qx[i][k] * qw[n][k] is an exact integer: |q| <= 7, so
// every product is an integer of magnitude <= 49 and, for K <= 32768, every
// partial sum stays below 2^24.  sm_103a has no integer tcgen05 MMA, so the
// codes ride on E4M3, which holds every integer in [-7, 7] exactly, through
// tcgen05.mma kind::f8f6f4 with fp32 accumulation in tensor memory; the
// integer accumulators come out exact as long as the fp32 sums are exact.
//
// CTA tile 128 (M) x 256 (N), K step 128 codes.  Warp roles (192 threads):
//   warp 4      TMA producer: packed A/B tiles (64 B x rows) into a 4-deep
//               ring of staging buffers;
//   warps 0-3   unpack nibbles to E4M3 bytes in the 128-byte-swizzled
//               K-major layout the MMA reads (2-deep ring), then run the
//               epilogue (TMEM -> registers -> scale, bias -> fp16/bf16);
//   warp 5      allocates TMEM (256 columns); one lane issues the MMAs.
// Every wait is bounded; see clq_device.cuh.
#include "clq_device.cuh"
#include "clq_kernels.h"

#include <cudaTypedefs.h>

namespace clq {

namespace {

constexpr int BM = 128;
constexpr int BN = 256;
constexpr int BK = 128;             // codes per K step
constexpr int BKP = BK / 2;         // packed bytes per row per K step
constexpr int SP = 4;               // packed staging stages
constexpr int SU = 2;               // unpacked operand stages
constexpr int A_P = BM * BKP;       // 8 KB
constexpr int B_P = BN * BKP;       // 16 KB
constexpr int A_U = BM * BK;        // 16 KB
constexpr int B_U = BN * BK;        // 32 KB
constexpr int TMEM_COLS = 256;
constexpr int THREADS = 192;

struct __align__(8) Barriers {
  uint64_t full_p[SP];
  uint64_t empty_p[SP];
  uint64_t full_u[SU];
  uint64_t empty_u[SU];
  uint64_t acc_full;
  uint32_t tmem_slot;
  int32_t abort;
};

constexpr size_t OFF_UA = 0;
constexpr size_t OFF_UB = OFF_UA + SU * A_U;
constexpr size_t OFF_PA = OFF_UB + SU * B_U;
constexpr size_t OFF_PB = OFF_PA + SP * A_P;
constexpr size_t OFF_COL = OFF_PB + SP * B_P;
constexpr size_t OFF_BAR = OFF_COL + 2 * BN * sizeof(float);
constexpr size_t SMEM_BYTES = OFF_BAR + sizeof(Barriers) + 1024;  // + alignment slack

__device__ __forceinline__ uint32_t pack2(uint16_t lo, uint16_t hi) {
  return static_cast<uint32_t>(lo) | (static_cast<uint32_t>(hi) << 16);
}

__device__ __forceinline__ uint32_t prmt(uint32_t a, uint32_t b, uint32_t c) {
  uint32_t d;
  asm("prmt.b32 %0, %1, %2, %3;" : "=r"(d) : "r"(a), "r"(b), "r"(c));
  return d;
}

// Eight 4-bit two's-complement codes (code j in nibble j) -> eight E4M3
// bytes.  Magnitude tables for the non-negative codes 0..7 and the negative
// codes -8..-1 are looked up with prmt on the low three bits of each nibble;
// the sign bit of each nibble, replicated to a byte mask by prmt's sign mode,
// selects between them.
__device__ __forceinline__ uint2 nibbles_to_e4m3(uint32_t w) {
  const uint32_t P0 = 0x44403800u, P1 = 0x4E4C4A48u;  // e4m3(0..7)
  const uint32_t N0 = 0xCACCCED0u, N1 = 0xB8C0C4C8u;  // e4m3(-8..-1)
  const uint32_t sel_lo = w & 0x7777u;
  const uint32_t sel_hi = (w >> 16) & 0x7777u;
  const uint32_t w4 = w << 4;
  const uint32_t m_lo = prmt(w4, w, 0xD9C8u);
  const uint32_t m_hi = prmt(w4, w, 0xFBEAu);
  const uint32_t p_lo = prmt(P0, P1, sel_lo), n_lo = prmt(N0, N1, sel_lo);
  const uint32_t p_hi = prmt(P0, P1, sel_hi), n_hi = prmt(N0, N1, sel_hi);
  return make_uint2((p_lo & ~m_lo) | (n_lo & m_lo), (p_hi & ~m_hi) | (n_hi & m_hi));
}

// Unpack `rows` x 64 packed bytes (row-major staging) into the 128-byte
// swizzled K-major E4M3 tile: row r, 16-byte chunk c lives at
// (r / 8) * 1024 + (r % 8) * 128 + ((c ^ (r % 8)) * 16).
template <int ROWS>
__device__ __forceinline__ void unpack_tile(const uint8_t* __restrict__ src,
                                            uint8_t* __restrict__ dst, int t) {
#pragma unroll
  for (int i = 0; i < ROWS * 4 / 128; ++i) {
    const int q = t + 128 * i;
    const int r = q >> 2;
    const int c = q & 3;
    const uint4 p = *reinterpret_cast<const uint4*>(src + r * BKP + c * 16);
    const uint2 e0 = nibbles_to_e4m3(p.x), e1 = nibbles_to_e4m3(p.y);
    const uint2 e2 = nibbles_to_e4m3(p.z), e3 = nibbles_to_e4m3(p.w);
    uint8_t* row = dst + (r >> 3) * 1024 + (r & 7) * 128;
    const int x = r & 7;
    *reinterpret_cast<uint4*>(row + (((2 * c) ^ x) << 4)) = make_uint4(e0.x, e0.y, e1.x, e1.y);
    *reinterpret_cast<uint4*>(row + (((2 * c + 1) ^ x) << 4)) =
        make_uint4(e2.x, e2.y, e3.x, e3.y);
  }
}

template <typename OutT>
__global__ void __launch_bounds__(THREADS, 1)
    w4a4_gemm_kernel(const __grid_constant__ CUtensorMap mapA,
                     const __grid_constant__ CUtensorMap mapB, GemmArgs g) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  Barriers* bars = reinterpret_cast<Barriers*>(smem + OFF_BAR);
  float* col_scale = reinterpret_cast<float*>(smem + OFF_COL);
  float* col_bias = col_scale + BN;
  volatile int32_t* abort = &bars->abort;

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int m0 = blockIdx.y * BM;
  const int n0 = blockIdx.x * BN;
  const int nk = (g.K + BK - 1) / BK;

  if (threadIdx.x == 0) {
    for (int s = 0; s < SP; ++s) {
      mbar_init(&bars->full_p[s], 1);
      mbar_init(&bars->empty_p[s], 128);
    }
    for (int s = 0; s < SU; ++s) {
      mbar_init(&bars->full_u[s], 128);
      mbar_init(&bars->empty_u[s], 1);
    }
    mbar_init(&bars->acc_full, 1);
    bars->abort = 0;
    fence_mbarrier_init();
  }
  if (warp == 4 && lane == 0) {
    prefetch_tensor_map(&mapA);
    prefetch_tensor_map(&mapB);
  }
  if (warp < 4) {
    for (int j = threadIdx.x; j < BN; j += 128) {
      const int col = n0 + j;
      float sc = 0.f, bi = 0.f;
      if (col < g.N) {
        sc = g.s_w[col] * g.inv_b;
        if (g.bias != nullptr)
          bi = Num<OutT>::to_f(static_cast<const uint16_t*>(g.bias)[col]);
      }
      col_scale[j] = sc;
      col_bias[j] = bi;
    }
  }
  if (warp == 5) {
    tmem_alloc(&bars->tmem_slot, TMEM_COLS);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = bars->tmem_slot;

  int issued = 0;  // producer: K steps whose copies were issued

  if (warp == 4) {
    if (lane == 0) {
      for (int kb = 0; kb < nk; ++kb) {
        const int s = kb % SP;
        const uint32_t ph = (kb / SP) & 1;
        if (!mbar_wait_bounded(&bars->empty_p[s], ph ^ 1, abort, g.status, kWaitLimitNs))
          break;
        mbar_arrive_expect_tx(&bars->full_p[s], A_P + B_P);
        tma_load_2d(smem + OFF_PA + s * A_P, &mapA, kb * BKP, m0, &bars->full_p[s]);
        tma_load_2d(smem + OFF_PB + s * B_P, &mapB, kb * BKP, n0, &bars->full_p[s]);
        ++issued;
      }
      // On an abort, let the copies already in flight land before exiting.
      if (*abort != 0) {
        for (int kb = std::max(0, issued - SP); kb < issued; ++kb)
          mbar_wait_bounded(&bars->full_p[kb % SP], (kb / SP) & 1, nullptr, nullptr,
                            10000000ull);
      }
    }
  } else if (warp == 5) {
    if (lane == 0) {
      constexpr uint32_t idesc = idesc_e4m3_f32(BM, BN);
      for (int kb = 0; kb < nk; ++kb) {
        const int u = kb % SU;
        const uint32_t ph = (kb / SU) & 1;
        if (!mbar_wait_bounded(&bars->full_u[u], ph, abort, g.status, kWaitLimitNs)) break;
        tc_fence_after();
        const uint32_t a0 = smem_addr(smem + OFF_UA + u * A_U);
        const uint32_t b0 = smem_addr(smem + OFF_UB + u * B_U);
#pragma unroll
        for (int k = 0; k < BK / 32; ++k)
          mma_e4m3(tmem, sw128_desc(a0 + k * 32), sw128_desc(b0 + k * 32), idesc,
                   (kb | k) != 0 ? 1u : 0u);
        mma_commit(&bars->empty_u[u]);
      }
      mma_commit(&bars->acc_full);
    }
  } else {
    const int t = threadIdx.x;  // 0..127
    bool ok = true;
    for (int kb = 0; kb < nk; ++kb) {
      const int s = kb % SP;
      const int u = kb % SU;
      if (!mbar_wait_bounded(&bars->full_p[s], (kb / SP) & 1, abort, g.status, kWaitLimitNs) ||
          !mbar_wait_bounded(&bars->empty_u[u], ((kb / SU) & 1) ^ 1, abort, g.status,
                             kWaitLimitNs)) {
        ok = false;
        break;
      }
      unpack_tile<BM>(smem + OFF_PA + s * A_P, smem + OFF_UA + u * A_U, t);
      unpack_tile<BN>(smem + OFF_PB + s * B_P, smem + OFF_UB + u * B_U, t);
      fence_proxy_async_smem();
      mbar_arrive(&bars->empty_p[s]);
      mbar_arrive(&bars->full_u[u]);
    }
    // ---- epilogue ----
    if (ok) ok = mbar_wait_bounded(&bars->acc_full, 0, abort, g.status, kWaitLimitNs);
    __syncwarp();
    ok = __all_sync(0xffffffffu, ok);
    if (ok) {
      tc_fence_after();
      const int row = m0 + t;
      const float sx = row < g.M ? g.s_x[row] : 0.f;
      const uint32_t lane_base = tmem + (static_cast<uint32_t>(warp * 32) << 16);
      OutT* yrow = static_cast<OutT*>(g.Y) + static_cast<size_t>(row) * g.N;
      const bool vec_ok = (g.N & 7) == 0;
#pragma unroll 1
      for (int c = 0; c < BN; c += 16) {
        if (n0 + c >= g.N) break;
        uint32_t r[16];
        tmem_ld16(lane_base + c, r);
        tmem_ld_wait();
        if (row < g.M) {
          uint16_t o[16];
#pragma unroll
          for (int j = 0; j < 16; ++j) {
            const float acc = __uint_as_float(r[j]);
            o[j] = Num<OutT>::from_f(fmaf(acc, sx * col_scale[c + j], col_bias[c + j]));
          }
          const int col0 = n0 + c;
          if (vec_ok && col0 + 16 <= g.N) {
            uint4* dst = reinterpret_cast<uint4*>(yrow + col0);
            dst[0] = make_uint4(pack2(o[0], o[1]), pack2(o[2], o[3]), pack2(o[4], o[5]),
                                pack2(o[6], o[7]));
            dst[1] = make_uint4(pack2(o[8], o[9]), pack2(o[10], o[11]), pack2(o[12], o[13]),
                                pack2(o[14], o[15]));
          } else {
            uint16_t* dst = reinterpret_cast<uint16_t*>(yrow);
#pragma unroll
            for (int j = 0; j < 16; ++j)
              if (col0 + j < g.N) dst[col0 + j] = o[j];
          }
          if (g.acc_dbg != nullptr) {
            int32_t* arow = g.acc_dbg + static_cast<size_t>(row) * g.N;
#pragma unroll
            for (int j = 0; j < 16; ++j)
              if (col0 + j < g.N) arow[col0 + j] = __float2int_rn(__uint_as_float(r[j]));
          }
        }
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 5) {
    tc_fence_after();
    // MMAs still in flight after an abort must finish before TMEM is freed.
    if (lane == 0 && *abort != 0)
      mbar_wait_bounded(&bars->acc_full, 0, nullptr, nullptr, 10000000ull);
    __syncwarp();
    tmem_dealloc(tmem, TMEM_COLS);
  }
}

}  // namespace

bool encode_tma_2d_u8(CUtensorMap* map, const void* base, uint64_t inner_bytes, uint64_t rows,
                      uint32_t box_inner, uint32_t box_rows) {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  if (fn == nullptr) {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000,
                                         cudaEnableDefault, &q) != cudaSuccess ||
        q != cudaDriverEntryPointSuccess || p == nullptr)
      return false;
    fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  }
  const cuuint64_t dims[2] = {inner_bytes, rows};
  const cuuint64_t strides[1] = {inner_bytes};
  const cuuint32_t box[2] = {box_inner, box_rows};
  const cuuint32_t estr[2] = {1, 1};
  const CUresult r = fn(map, CU_TENSOR_MAP_DATA_TYPE_UINT8, 2, const_cast<void*>(base), dims,
                        strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                        CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                        CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

cudaError_t launch_w4a4_gemm(const uint8_t* Xq, const uint8_t* Wq, const GemmArgs& g,
                             int out_dtype, cudaStream_t st) {
  CUtensorMap mapA, mapB;
  const uint64_t kb = static_cast<uint64_t>(g.K) / 2;
  if (!encode_tma_2d_u8(&mapA, Xq, kb, static_cast<uint64_t>(g.M), BKP, BM) ||
      !encode_tma_2d_u8(&mapB, Wq, kb, static_cast<uint64_t>(g.N), BKP, BN))
    return cudaErrorInvalidValue;
  const dim3 grid((g.N + BN - 1) / BN, (g.M + BM - 1) / BM);
  if (out_dtype == CLQ_F16) {
    auto k = w4a4_gemm_kernel<__half>;
    cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         static_cast<int>(SMEM_BYTES));
    if (e != cudaSuccess) return e;
    k<<<grid, THREADS, SMEM_BYTES, st>>>(mapA, mapB, g);
  } else {
    auto k = w4a4_gemm_kernel<__nv_bfloat16>;
    cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         static_cast<int>(SMEM_BYTES));
    if (e != cudaSuccess) return e;
    k<<<grid, THREADS, SMEM_BYTES, st>>>(mapA, mapB, g);
  }
  return cudaGetLastError();
}

// ------------------------------------------------------ bounded-wait test ---
namespace {
__global__ void wait_selftest_kernel(uint64_t timeout_ns, int32_t* status) {
  __shared__ __align__(8) uint64_t bar;
  __shared__ int32_t abort;
  if (threadIdx.x == 0) {
    mbar_init(&bar, 1);
    abort = 0;
    fence_mbarrier_init();
  }
  __syncthreads();
  if (threadIdx.x == 0) mbar_wait_bounded(&bar, 0, &abort, status, timeout_ns);
  __syncthreads();
}
}  // namespace

cudaError_t launch_wait_selftest(uint64_t timeout_ns, int32_t* status, cudaStream_t st) {
  wait_selftest_kernel<<<1, 32, 0, st>>>(timeout_ns, status);
  return cudaGetLastError();
}

}  // namespace clq
