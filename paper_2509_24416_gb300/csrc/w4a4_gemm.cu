// Standalone W4A4 GEMM kernel (pipeline in gemm_pipeline.cuh), the weight
// expansion kernel, TMA descriptor helpers and the bounded-wait self test.
#include "gemm_pipeline.cuh"

#include <cudaTypedefs.h>

#include <atomic>
#include <map>
#include <mutex>
#include <set>
#include <tuple>

namespace clq {

namespace {

using namespace gemm;

// W8A8 tiles: three accumulators of 128 columns fill one TMEM allocation.
constexpr int kSepBN = 128;

template <bool APACK, bool BPACK, int BNT, int PA, int PB, bool SEP = false>
constexpr size_t smem_bytes() {
  return Cfg<APACK, BPACK, BNT, PA, PB, 0, MAX_STAGES, SEP>::BYTES + 1024;  // + alignment slack
}

// PA / PB = 2: the activation / weight codes are 8-bit, as two E4M3 planes
// (mapA2 / mapB2 the second plane).
template <typename OutT, bool APACK, bool BPACK, int BNT, int PA, int PB, bool ASYM, bool F6,
          bool SEP>
__global__ void __launch_bounds__((Cfg<APACK, BPACK, BNT, PA, PB>::THREADS), 1)
    w4a4_gemm_kernel(const __grid_constant__ CUtensorMap mapA,
                     const __grid_constant__ CUtensorMap mapB,
                     const __grid_constant__ CUtensorMap mapY,
                     const __grid_constant__ CUtensorMap mapA2,
                     const __grid_constant__ CUtensorMap mapB2, GemmArgs g, int use_tma_store) {
  extern __shared__ uint8_t smem_raw[];
  __shared__ Barriers bars;
  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  setup<APACK, BPACK, BNT, PA, PB, 0, MAX_STAGES, SEP>(&bars);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = bars.tmem_slot;
  // The tensor maps are kernel parameters, not outputs of the previous kernel:
  // fetch them while it finishes (measured +0.25 % on the PixArt step).
  if (threadIdx.x == WARP_TMA * 32) {
    prefetch_tensor_map(&mapA);
    prefetch_tensor_map(&mapB);
    if (use_tma_store) prefetch_tensor_map(&mapY);
    // The weight boxes of this CTA's first pipeline stages into L2 (a hint:
    // it changes no value the copies after the wait read).
    using C = Cfg<APACK, BPACK, BNT, PA, PB, 0, MAX_STAGES, SEP>;
    const int tiles_n = (g.N + BNT - 1) / BNT;
    const int tiles = ((g.M + BM - 1) / BM) * tiles_n;
    if (!BPACK && static_cast<int>(blockIdx.x) < tiles) {
      const int n0 = (static_cast<int>(blockIdx.x) % tiles_n) * BNT;
      const int nk = (g.K + BK - 1) / BK;
      for (int kb = 0; kb < C::S && kb < nk; ++kb) {
        tma_prefetch_2d(&mapB, kb * BK, n0);
        if (PB == 2) tma_prefetch_2d(&mapB2, kb * BK, n0);
      }
    }
  }
  // Barriers and TMEM are set up; global inputs are read only from here on.
  pdl_wait();
  pdl_launch_dependents();
  const Maps maps{&mapA, &mapB, use_tma_store ? &mapY : nullptr, &mapA2, &mapB2};
  pipeline<OutT, APACK, BPACK, BNT, true, PA, PB, ASYM, 0, MAX_STAGES, F6, SEP>(
      maps, g, smem, &bars, tmem, nullptr);
  tc_fence_before();
  __syncthreads();
  teardown(tmem, Cfg<APACK, BPACK, BNT, PA, PB, 0, MAX_STAGES, SEP>::TMEM);
}

// Packed INT4 weights -> E4M3 execution layout (one code per byte, the byte
// is the E4M3 encoding of the integer code).  16 packed bytes per thread.
__global__ void expand_weights_kernel(const uint4* __restrict__ src, uint4* __restrict__ dst,
                                      size_t n16) {
  for (size_t i = blockIdx.x * static_cast<size_t>(blockDim.x) + threadIdx.x; i < n16;
       i += static_cast<size_t>(gridDim.x) * blockDim.x) {
    const uint4 p = src[i];
    const uint2 e0 = nibbles_to_e4m3(p.x), e1 = nibbles_to_e4m3(p.y);
    const uint2 e2 = nibbles_to_e4m3(p.z), e3 = nibbles_to_e4m3(p.w);
    dst[2 * i] = make_uint4(e0.x, e0.y, e1.x, e1.y);
    dst[2 * i + 1] = make_uint4(e2.x, e2.y, e3.x, e3.y);
  }
}

// Value of an E4M3 byte that holds an integer code (exact): sign, exponent
// with bias 7, three mantissa bits.
__device__ __forceinline__ int e4m3_int(uint32_t byte) {
  const int e = (byte >> 3) & 0xF;
  const int m = byte & 0x7;
  const float v = e == 0 ? 0.f : ldexpf(static_cast<float>(8 + m), e - 10);
  const int i = static_cast<int>(v);
  return (byte & 0x80u) ? -i : i;
}

// Value of the 6-bit E2M3 field f (sign bit 5, exponent bits 4-3 with bias 1,
// three mantissa bits) times 8, exact: an integer code q gives 8 q.
__device__ __forceinline__ int e2m3_times8(uint32_t f) {
  const int e = (f >> 3) & 0x3;
  const int m = f & 0x7;
  const int v = e == 0 ? m : (8 + m) << (e - 1);
  return (f & 0x20u) ? -v : v;
}

// The 16 codes of group g (codes 16 g .. 16 g + 15) of a row in a 4-bit layout
// (packed nibbles, E4M3 bytes or E2M3 fields), as integers; false if a field
// holds no integer (only E2M3 and E4M3 fields can).
__device__ __forceinline__ bool decode_group(const uint8_t* __restrict__ row, int codes, int g,
                                             int (&c)[16]) {
  bool ok = true;
  if (codes == CLQ_CODES_INT4_PACKED) {
    const uint8_t* p = row + 8 * g;
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      const int lo = p[j] & 0xF, hi = p[j] >> 4;
      c[2 * j] = lo >= 8 ? lo - 16 : lo;
      c[2 * j + 1] = hi >= 8 ? hi - 16 : hi;
    }
  } else if (codes == CLQ_CODES_E2M3) {
    const uint8_t* p = row + 12 * g;
    uint64_t lo = 0, hi = 0;  // the 96-bit group, little-endian
#pragma unroll
    for (int j = 0; j < 8; ++j) lo |= static_cast<uint64_t>(p[j]) << (8 * j);
#pragma unroll
    for (int j = 0; j < 4; ++j) hi |= static_cast<uint64_t>(p[8 + j]) << (8 * j);
#pragma unroll
    for (int i = 0; i < 16; ++i) {
      const int bit = 6 * i;
      const uint32_t f = static_cast<uint32_t>(
          (bit < 64 ? (lo >> bit) | (bit > 58 ? hi << (64 - bit) : 0ull) : hi >> (bit - 64)) &
          0x3Full);
      const int v8 = e2m3_times8(f);
      ok &= (v8 & 7) == 0;
      c[i] = v8 / 8;
    }
  } else {
    const uint8_t* p = row + 16 * g;
#pragma unroll
    for (int j = 0; j < 16; ++j) c[j] = e4m3_int(p[j]);
  }
  return ok;
}

// Bytes of one row of K codes in a layout.
__host__ __device__ __forceinline__ size_t codes_row_bytes(int codes, int K) {
  return codes == CLQ_CODES_INT4_PACKED ? static_cast<size_t>(K) / 2
         : codes == CLQ_CODES_E2M3      ? static_cast<size_t>(K) / 4 * 3
         : codes == CLQ_CODES_E4M3_SPLIT ? 2 * static_cast<size_t>(K)
                                         : static_cast<size_t>(K);
}

// One group of 16 integer codes in [-7, 7] into a 4-bit layout.
__device__ __forceinline__ void encode_group(uint8_t* __restrict__ row, int codes, int g,
                                             const int (&c)[16]) {
  if (codes == CLQ_CODES_INT4_PACKED) {
#pragma unroll
    for (int j = 0; j < 8; ++j)
      row[8 * g + j] = static_cast<uint8_t>((c[2 * j] & 0xF) | ((c[2 * j + 1] & 0xF) << 4));
  } else if (codes == CLQ_CODES_E2M3) {
    // E2M3 encodings of 0..7: exponent 0 for 0, else 1..3, mantissa in eighths
    constexpr uint8_t kMag[8] = {0x00, 0x08, 0x10, 0x14, 0x18, 0x1A, 0x1C, 0x1E};
    uint64_t lo = 0, hi = 0;
#pragma unroll
    for (int i = 0; i < 16; ++i) {
      const uint64_t f = kMag[c[i] < 0 ? -c[i] : c[i]] | (c[i] < 0 ? 0x20u : 0u);
      const int bit = 6 * i;
      if (bit < 64) {
        lo |= f << bit;
        if (bit + 6 > 64) hi |= f >> (64 - bit);
      } else {
        hi |= f << (bit - 64);
      }
    }
#pragma unroll
    for (int j = 0; j < 8; ++j) row[12 * g + j] = static_cast<uint8_t>(lo >> (8 * j));
#pragma unroll
    for (int j = 0; j < 4; ++j) row[12 * g + 8 + j] = static_cast<uint8_t>(hi >> (8 * j));
  } else {
    // E4M3 encodings of 0..7 (exponent bias 7), sign bit 7
    constexpr uint8_t kMag[8] = {0x00, 0x38, 0x40, 0x44, 0x48, 0x4A, 0x4C, 0x4E};
#pragma unroll
    for (int j = 0; j < 16; ++j)
      row[16 * g + j] = kMag[c[j] < 0 ? -c[j] : c[j]] | (c[j] < 0 ? 0x80u : 0u);
  }
}

// Code array in one 4-bit layout -> another, one thread a group of 16 codes.
// A code outside [-7, 7] (packed -8) or a field that holds no integer is
// written as 0 and reported.
__global__ void convert_codes_kernel(const uint8_t* __restrict__ src, int src_codes,
                                     uint8_t* __restrict__ dst, int dst_codes, int rows, int K,
                                     int32_t* status) {
  const int groups = K / 16;
  const size_t n = static_cast<size_t>(rows) * groups;
  const size_t sb = codes_row_bytes(src_codes, K), db = codes_row_bytes(dst_codes, K);
  for (size_t i = blockIdx.x * static_cast<size_t>(blockDim.x) + threadIdx.x; i < n;
       i += static_cast<size_t>(gridDim.x) * blockDim.x) {
    const size_t r = i / groups;
    const int g = static_cast<int>(i - r * groups);
    int c[16];
    bool ok = decode_group(src + r * sb, src_codes, g, c);
#pragma unroll
    for (int j = 0; j < 16; ++j) {
      const bool in = c[j] >= -7 && c[j] <= 7;
      ok &= in;
      if (!in) c[j] = 0;
    }
    if (!ok) record_status(status, CLQ_ERR_DEVICE_CODE);
    encode_group(dst + r * db, dst_codes, g, c);
  }
}

// sum_k q[n][k] of each row of a code array (any layout), one warp a row.
__global__ void code_sums_kernel(const uint8_t* __restrict__ W, int codes, int N, int K,
                                 float* __restrict__ wsum) {
  const int warp = (blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  if (warp >= N) return;
  if (codes == CLQ_CODES_E2M3) {
    const uint8_t* row = W + static_cast<size_t>(warp) * codes_row_bytes(codes, K);
    int acc = 0;
    for (int gi = lane; gi < K / 16; gi += 32) {
      int c[16];
      decode_group(row, codes, gi, c);
#pragma unroll
      for (int j = 0; j < 16; ++j) acc += c[j];
    }
    for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
    if (lane == 0) wsum[warp] = static_cast<float>(acc);
    return;
  }
  const int width = codes == CLQ_CODES_INT4_PACKED ? K / 2
                    : codes == CLQ_CODES_E4M3_SPLIT ? 2 * K : K;
  const uint4* row = reinterpret_cast<const uint4*>(W + static_cast<size_t>(warp) * width);
  int acc = 0;
  for (int i = lane; i < width / 16; i += 32) {
    const uint4 p = __ldg(row + i);
    const uint32_t w[4] = {p.x, p.y, p.z, p.w};
#pragma unroll
    for (int j = 0; j < 4; ++j) {
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        const uint32_t byte = (w[j] >> (8 * k)) & 0xFFu;
        if (codes == CLQ_CODES_INT4_PACKED) {
          const int lo = static_cast<int>(byte & 0xFu), hi = static_cast<int>(byte >> 4);
          acc += (lo >= 8 ? lo - 16 : lo) + (hi >= 8 ? hi - 16 : hi);
        } else {
          acc += e4m3_int(byte);
        }
      }
    }
  }
  for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
  if (lane == 0) wsum[warp] = static_cast<float>(acc);
}

}  // namespace

cudaError_t launch_code_sums(const uint8_t* W, int codes, int N, int K, float* wsum,
                             cudaStream_t st) {
  const int blocks = (N + 7) / 8;
  code_sums_kernel<<<blocks, 256, 0, st>>>(W, codes, N, K, wsum);
  return cudaGetLastError();
}

bool encode_tma_2d_strided(CUtensorMap* map, CUtensorMapDataType dt, uint32_t esize,
                           const void* base, uint64_t inner, uint64_t rows,
                           uint64_t row_stride_bytes, uint32_t box_inner, uint32_t box_rows,
                           CUtensorMapSwizzle swz) {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  if (fn == nullptr) {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                         &q) != cudaSuccess ||
        q != cudaDriverEntryPointSuccess || p == nullptr)
      return false;
    fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  }
  const cuuint64_t dims[2] = {inner, rows};
  const cuuint64_t strides[1] = {row_stride_bytes};
  const cuuint32_t box[2] = {box_inner, box_rows};
  const cuuint32_t estr[2] = {1, 1};
  const CUresult r = fn(map, dt, 2, const_cast<void*>(base), dims, strides, box, estr,
                        CU_TENSOR_MAP_INTERLEAVE_NONE, swz, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                        CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

bool encode_tma_2d(CUtensorMap* map, CUtensorMapDataType dt, uint32_t esize, const void* base,
                   uint64_t inner, uint64_t rows, uint32_t box_inner, uint32_t box_rows,
                   CUtensorMapSwizzle swz) {
  return encode_tma_2d_strided(map, dt, esize, base, inner, rows, inner * esize, box_inner,
                               box_rows, swz);
}


bool encode_tma_2d_u8(CUtensorMap* map, const void* base, uint64_t inner_bytes, uint64_t rows,
                      uint32_t box_inner, uint32_t box_rows) {
  return encode_tma_2d(map, CU_TENSOR_MAP_DATA_TYPE_UINT8, 1, base, inner_bytes, rows, box_inner,
                       box_rows, CU_TENSOR_MAP_SWIZZLE_NONE);
}

bool encode_tma_out_tile(CUtensorMap* map, void* Y, int M, int N) {
  return encode_tma_2d(map, CU_TENSOR_MAP_DATA_TYPE_UINT16, 2, Y, static_cast<uint64_t>(N),
                       static_cast<uint64_t>(M), EPI_COLS, EPI_ROWS, CU_TENSOR_MAP_SWIZZLE_64B);
}

int sm_count() {
  static std::atomic<int> cached[64];
  int dev = 0, sms = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 0;
  sms = cached[dev].load(std::memory_order_relaxed);
  if (sms > 0) return sms;
  if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return 0;
  cached[dev].store(sms, std::memory_order_relaxed);
  return sms;
}

cudaError_t kernel_setup(const void* func, size_t smem, int threads, int* per_sm) {
  static std::mutex mu;
  static std::map<std::tuple<const void*, int, size_t, int>, int> occupancy;
  static std::set<std::pair<const void*, int>> raised;
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  std::lock_guard<std::mutex> lock(mu);
  if (raised.count({func, dev}) == 0) {
    int optin = 0;
    e = cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev);
    if (e != cudaSuccess) return e;
    cudaFuncAttributes fa;
    e = cudaFuncGetAttributes(&fa, func);
    if (e != cudaSuccess) return e;
    e = cudaFuncSetAttribute(func, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             optin - static_cast<int>(fa.sharedSizeBytes));
    if (e != cudaSuccess) return e;
    raised.insert({func, dev});
  }
  if (per_sm != nullptr) {
    const auto key = std::make_tuple(func, dev, smem, threads);
    auto it = occupancy.find(key);
    if (it == occupancy.end()) {
      int n = 0;
      e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, func, threads, smem);
      if (e != cudaSuccess) return e;
      it = occupancy.emplace(key, n).first;
    }
    *per_sm = it->second;
  }
  return cudaSuccess;
}

namespace {

struct MapSet {
  CUtensorMap A, B, Y, A2, B2;
};

template <typename OutT, bool APACK, bool BPACK, int BNT, int PA = 1, int PB = 1,
          bool ASYM = false, bool F6 = false>
cudaError_t launch_gemm_t(const MapSet& m, const GemmArgs& g, int use_tma_store, int grid,
                          cudaStream_t st) {
  constexpr bool SEP = PA == 2 && PB == 2;  // W8A8: exact plane accumulators
  auto k = w4a4_gemm_kernel<OutT, APACK, BPACK, BNT, PA, PB, ASYM, F6, SEP>;
  constexpr size_t smem = smem_bytes<APACK, BPACK, BNT, PA, PB, SEP>();
  constexpr int threads = Cfg<APACK, BPACK, BNT, PA, PB>::THREADS;
  cudaError_t e = kernel_setup(reinterpret_cast<const void*>(k), smem, threads, nullptr);
  if (e != cudaSuccess) return e;
  return launch_pdl(k, grid, threads, smem, st, m.A, m.B, m.Y, m.A2, m.B2, g, use_tma_store);
}

template <typename OutT>
cudaError_t launch_gemm_dt(const MapSet& m, const GemmArgs& g, int x_codes, int w_codes, int bn,
                           int use_tma_store, int grid, cudaStream_t st) {
  const bool apack = x_codes == CLQ_CODES_INT4_PACKED;
  const bool bpack = w_codes == CLQ_CODES_INT4_PACKED;
  if (x_codes == CLQ_CODES_E2M3) {  // both operands E2M3 (checked by the caller)
    if (bn == 192)
      return launch_gemm_t<OutT, false, false, 192, 1, 1, false, true>(m, g, use_tma_store, grid,
                                                                        st);
    return launch_gemm_t<OutT, false, false, BN, 1, 1, false, true>(m, g, use_tma_store, grid, st);
  }
  if (g.lo != nullptr) {  // asymmetric activations: E4M3 / split operands only
    if (x_codes == CLQ_CODES_E4M3_SPLIT)
      return w_codes == CLQ_CODES_E4M3_SPLIT
                 ? launch_gemm_t<OutT, false, false, kSepBN, 2, 2, true>(m, g, use_tma_store,
                                                                         grid, st)
                 : launch_gemm_t<OutT, false, false, BN, 2, 1, true>(m, g, use_tma_store, grid,
                                                                     st);
    return launch_gemm_t<OutT, false, false, BN, 1, 1, true>(m, g, use_tma_store, grid, st);
  }
  if (x_codes == CLQ_CODES_E4M3_SPLIT)
    return w_codes == CLQ_CODES_E4M3_SPLIT
               ? launch_gemm_t<OutT, false, false, kSepBN, 2, 2>(m, g, use_tma_store, grid, st)
               : launch_gemm_t<OutT, false, false, BN, 2, 1>(m, g, use_tma_store, grid, st);
  if (apack)
    return bpack ? launch_gemm_t<OutT, true, true, BN>(m, g, use_tma_store, grid, st)
                 : launch_gemm_t<OutT, true, false, BN>(m, g, use_tma_store, grid, st);
  if (bpack) return launch_gemm_t<OutT, false, true, BN>(m, g, use_tma_store, grid, st);
  if (bn == 192) return launch_gemm_t<OutT, false, false, 192>(m, g, use_tma_store, grid, st);
  return launch_gemm_t<OutT, false, false, BN>(m, g, use_tma_store, grid, st);
}

}  // namespace

// TMA map of a code array (rows x K codes) in any layout: packed boxes of 64
// bytes x box_rows (no swizzle, staged for unpacking), E4M3 boxes of 128
// bytes x box_rows with the 128-byte swizzle (MMA operand), or E2M3 boxes of
// 128 codes x box_rows (96 bytes a row in global memory, 128 in shared
// memory, 128-byte swizzle; K a multiple of 128).  For the split
// layout ([rows][2][K]) the map covers plane `plane` of every row (row stride
// 2K bytes); for the others `plane` must be 0.
bool encode_codes_map(CUtensorMap* map, const uint8_t* base, int codes, int rows, int K,
                      int box_rows, int plane) {
  if (codes == CLQ_CODES_E2M3)  // 16 codes in 12 bytes, each group padded to 16 in smem
    return encode_tma_2d_strided(map, CU_TENSOR_MAP_DATA_TYPE_16U6_ALIGN16B, 1, base,
                                 static_cast<uint64_t>(K), static_cast<uint64_t>(rows),
                                 static_cast<uint64_t>(K) / 4 * 3, BK, box_rows,
                                 CU_TENSOR_MAP_SWIZZLE_128B);
  if (codes == CLQ_CODES_INT4_PACKED)
    return encode_tma_2d_u8(map, base, static_cast<uint64_t>(K) / 2, static_cast<uint64_t>(rows),
                            BKP, box_rows);
  const bool split = codes == CLQ_CODES_E4M3_SPLIT;
  return encode_tma_2d_strided(map, CU_TENSOR_MAP_DATA_TYPE_UINT8, 1,
                               base + (split ? static_cast<size_t>(plane) * K : 0),
                               static_cast<uint64_t>(K), static_cast<uint64_t>(rows),
                               static_cast<uint64_t>(K) * (split ? 2 : 1), BK, box_rows,
                               CU_TENSOR_MAP_SWIZZLE_128B);
}

// Tile width of the E4M3 x E4M3 GEMM: an SM's intake from L2 bounds the
// kernel, so a tile costs about its operand bytes per K step (A 16 KB + B
// BN/8 KB), and the CTAs walk ceil(tiles / SMs) rounds.  256 wins unless 192
// splits N into whole tiles with no more rounds (N = 1152: 6 x 192 instead of
// 4.5 x 256).  128 measured slower everywhere.
int gemm_tile_n(int M, int N, int sms) {
  const long mt = (M + BM - 1) / BM;
  auto cost = [&](int w) {
    const long rounds = (mt * ((N + w - 1) / w) + sms - 1) / sms;
    return rounds * (16.0 + w / 8.0);
  };
  return cost(192) < cost(256) ? 192 : BN;
}

cudaError_t launch_w4a4_gemm(const uint8_t* Xq, int x_codes, const uint8_t* W, int w_codes,
                             const GemmArgs& g, int out_dtype, cudaStream_t st) {
  const int sms = sm_count();
  if (sms <= 0) return cudaErrorInvalidDevice;
  const bool apack = x_codes == CLQ_CODES_INT4_PACKED;
  const bool bpack = w_codes == CLQ_CODES_INT4_PACKED;
  const bool split = x_codes == CLQ_CODES_E4M3_SPLIT || w_codes == CLQ_CODES_E4M3_SPLIT;
  // The tile-width model weighs operand bytes per K step; E2M3 scales both
  // widths' bytes by the same 3/4, so the choice is the same.
  const bool w8a8 = x_codes == CLQ_CODES_E4M3_SPLIT && w_codes == CLQ_CODES_E4M3_SPLIT;
  const int bn = w8a8 ? kSepBN
                      : (!apack && !bpack && !split && g.lo == nullptr) ? gemm_tile_n(g.M, g.N, sms)
                                                                         : BN;
  MapSet m;
  if (!encode_codes_map(&m.A, Xq, x_codes, g.M, g.K, BM, 0) ||
      !encode_codes_map(&m.B, W, w_codes, g.N, g.K, bn, 0))
    return cudaErrorInvalidValue;
  m.A2 = m.A;  // unused unless split
  m.B2 = m.B;
  if (x_codes == CLQ_CODES_E4M3_SPLIT && !encode_codes_map(&m.A2, Xq, x_codes, g.M, g.K, BM, 1))
    return cudaErrorInvalidValue;
  if (w_codes == CLQ_CODES_E4M3_SPLIT && !encode_codes_map(&m.B2, W, w_codes, g.N, g.K, bn, 1))
    return cudaErrorInvalidValue;
  const int use_tma_store = (g.N % 8 == 0) ? 1 : 0;
  if (use_tma_store) {
    if (!encode_tma_out_tile(&m.Y, g.Y, g.M, g.N)) return cudaErrorInvalidValue;
  } else {
    m.Y = m.A;  // unused
  }
  const int tiles = ((g.M + BM - 1) / BM) * ((g.N + bn - 1) / bn);
  const int grid = std::min(tiles, sms);
  if (out_dtype == CLQ_F16)
    return launch_gemm_dt<__half>(m, g, x_codes, w_codes, bn, use_tma_store, grid, st);
  return launch_gemm_dt<__nv_bfloat16>(m, g, x_codes, w_codes, bn, use_tma_store, grid, st);
}

cudaError_t launch_convert_codes(const uint8_t* src, int src_codes, uint8_t* dst, int dst_codes,
                                 int rows, int K, int32_t* status, cudaStream_t st) {
  const size_t n = static_cast<size_t>(rows) * (K / 16);
  const int sms = sm_count();
  if (sms <= 0) return cudaErrorInvalidDevice;
  const int blocks = static_cast<int>(std::min<size_t>((n + 255) / 256, 8u * sms));
  convert_codes_kernel<<<std::max(blocks, 1), 256, 0, st>>>(src, src_codes, dst, dst_codes, rows,
                                                            K, status);
  return cudaGetLastError();
}

cudaError_t launch_expand_weights(const uint8_t* Wq, int N, int K, uint8_t* We, cudaStream_t st) {
  const size_t n16 = static_cast<size_t>(N) * (K / 2) / 16;
  const int sms = sm_count();
  if (sms <= 0) return cudaErrorInvalidDevice;
  const int blocks = static_cast<int>(std::min<size_t>((n16 + 255) / 256, 8u * sms));
  expand_weights_kernel<<<std::max(blocks, 1), 256, 0, st>>>(
      reinterpret_cast<const uint4*>(Wq), reinterpret_cast<uint4*>(We), n16);
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
