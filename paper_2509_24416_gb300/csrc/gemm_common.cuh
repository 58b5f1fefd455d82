// Pieces shared by the W4A4 GEMM and the fused rotate-quant + GEMM kernels:
// tile shape, nibble -> E4M3 unpacking into the tcgen05 operand layout, and
// the TMEM -> fp16/bf16 epilogue with TMA stores.
#pragma once

#include "clq_device.cuh"

namespace clq {
namespace gemm {

constexpr int BM = 128;           // rows of A (tokens) per tile
constexpr int BN = 256;           // rows of B (output channels) per tile (widest)
constexpr int BK = 128;           // codes per K step = one 128-byte swizzle row
constexpr int BKP = BK / 2;       // packed bytes per row per K step
constexpr int A_U = BM * BK;      // 16 KB unpacked A stage
constexpr int B_U = BN * BK;      // 32 KB unpacked B stage
constexpr int A_P = BM * BKP;     // 8 KB packed A stage
constexpr int B_P = BN * BKP;     // 16 KB packed B stage
constexpr int EPI_COLS = 32;      // output columns per epilogue store
constexpr int EPI_ROWS = 32;      // rows per store: one warp's TMEM lanes
constexpr int EPI_BYTES = EPI_ROWS * EPI_COLS * 2;  // 2 KB staging buffer
constexpr int EPI_TOTAL = 8 * EPI_BYTES;            // 4 warps x 2 or 8 warps x 1
constexpr int TMEM_COLS = 512;    // two 128 x 256 fp32 accumulators
constexpr uint32_t kEpiBarrier = 1;  // named barrier id of the epilogue warps

__device__ __forceinline__ uint32_t prmt(uint32_t a, uint32_t b, uint32_t c) {
  uint32_t d;
  asm("prmt.b32 %0, %1, %2, %3;" : "=r"(d) : "r"(a), "r"(b), "r"(c));
  return d;
}

__device__ __forceinline__ uint32_t pack2(uint16_t lo, uint16_t hi) {
  return static_cast<uint32_t>(lo) | (static_cast<uint32_t>(hi) << 16);
}

__device__ __forceinline__ void named_bar_sync(uint32_t id, uint32_t threads) {
  asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(threads) : "memory");
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

// Byte offset of 16-byte chunk c (0..7) of row r in a K-major E4M3 operand
// tile with the 128-byte swizzle: 8-row atoms of 1024 bytes.
__device__ __forceinline__ uint32_t sw128_offset(int r, int c) {
  return static_cast<uint32_t>((r >> 3) * 1024 + (r & 7) * 128 + ((c ^ (r & 7)) << 4));
}

// Unpack ROWS x 64 packed bytes (row-major staging) into the swizzled E4M3
// tile, NT threads cooperating (thread index t).
template <int ROWS, int NT>
__device__ __forceinline__ void unpack_rows(const uint8_t* __restrict__ src,
                                            uint8_t* __restrict__ dst, int t) {
#pragma unroll
  for (int i = 0; i < ROWS * 4 / NT; ++i) {
    const int q = t + NT * i;
    const int r = q >> 2;
    const int c = q & 3;
    const uint4 p = *reinterpret_cast<const uint4*>(src + r * BKP + c * 16);
    const uint2 e0 = nibbles_to_e4m3(p.x), e1 = nibbles_to_e4m3(p.y);
    const uint2 e2 = nibbles_to_e4m3(p.z), e3 = nibbles_to_e4m3(p.w);
    *reinterpret_cast<uint4*>(dst + sw128_offset(r, 2 * c)) = make_uint4(e0.x, e0.y, e1.x, e1.y);
    *reinterpret_cast<uint4*>(dst + sw128_offset(r, 2 * c + 1)) =
        make_uint4(e2.x, e2.y, e3.x, e3.y);
  }
}

// 32 lanes x 32 bit, 32 consecutive columns per thread.
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, uint32_t (&r)[32]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
      "{%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,"
      "%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
        "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]),
        "=r"(r[13]), "=r"(r[14]), "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]),
        "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]),
        "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]),
        "=r"(r[31])
      : "r"(taddr));
}

__device__ __forceinline__ void tma_store_2d(const CUtensorMap* map, const void* smem_src,
                                             int32_t x, int32_t y) {
  asm volatile(
      "cp.async.bulk.tensor.2d.global.shared::cta.tile.bulk_group [%0, {%2, %3}], [%1];" ::"l"(
          reinterpret_cast<uint64_t>(map)),
      "r"(smem_addr(smem_src)), "r"(x), "r"(y)
      : "memory");
}

__device__ __forceinline__ void bulk_commit() {
  asm volatile("cp.async.bulk.commit_group;" ::: "memory");
}

template <int N>
__device__ __forceinline__ void bulk_wait_read() {
  asm volatile("cp.async.bulk.wait_group.read %0;" ::"n"(N) : "memory");
}

__device__ __forceinline__ void bulk_wait_all() {
  asm volatile("cp.async.bulk.wait_group 0;" ::: "memory");
}

// Wait for this thread's outstanding tcgen05.ld and make every register of
// r depend on that wait, so that no use of r is scheduled before it.
__device__ __forceinline__ void tmem_ld_wait_tie(uint32_t (&r)[32]) {
  tmem_ld_wait();
#pragma unroll
  for (int i = 0; i < 32; ++i) asm volatile("" : "+r"(r[i]));
}

// One 32-row x 32-column block of the epilogue (the block at tile column c):
// y = acc * s_x[row] * s_w[col] / b + bias[col], rounded to OutT, where
// col_scale / col_bias hold s_w / b and bias for the tile's columns.  With a
// TMA map for Y the block goes through one of the warp's NBUF 64-byte-swizzled
// staging buffers and one bulk tensor store issued by lane 0; otherwise (N not
// a multiple of 8) each lane stores its row directly.
// ASYM (asymmetric activation codes, centered): s_x[row] is the row's step
// delta, zm the value of code 0, col_zw holds sum_k q_w[col][k] * s_w / b,
// and y = acc * delta * s_w / b + zm * col_zw + bias.
template <typename OutT, int NBUF, bool ASYM = false>
__device__ __forceinline__ void epilogue_block(const uint32_t (&r)[32], int c, int quarter,
                                               int lane, int m0, int n0, int M, int N,
                                               float sx, const float* col_scale,
                                               const float* col_bias, float zm,
                                               const float* col_zw, uint8_t* staging,
                                               const CUtensorMap* mapY, void* Y,
                                               int32_t* acc_dbg, int& store_count) {
  const int row = m0 + quarter * 32 + lane;
  uint32_t o[16];
  const float2 sx2 = make_float2(sx, sx);
#pragma unroll
  for (int j = 0; j < 8; ++j) {
    const float4 cs = *reinterpret_cast<const float4*>(col_scale + c + 4 * j);
    float4 cb = *reinterpret_cast<const float4*>(col_bias + c + 4 * j);
    if constexpr (ASYM) {
      const float4 cz = *reinterpret_cast<const float4*>(col_zw + c + 4 * j);
      const float2 zm2 = make_float2(zm, zm);
      const float2 b0 = __ffma2_rn(zm2, make_float2(cz.x, cz.y), make_float2(cb.x, cb.y));
      const float2 b1 = __ffma2_rn(zm2, make_float2(cz.z, cz.w), make_float2(cb.z, cb.w));
      cb = make_float4(b0.x, b0.y, b1.x, b1.y);
    }
    const float2 a0 = make_float2(__uint_as_float(r[4 * j]), __uint_as_float(r[4 * j + 1]));
    const float2 a1 = make_float2(__uint_as_float(r[4 * j + 2]), __uint_as_float(r[4 * j + 3]));
    const float2 y0 =
        __ffma2_rn(a0, __fmul2_rn(sx2, make_float2(cs.x, cs.y)), make_float2(cb.x, cb.y));
    const float2 y1 =
        __ffma2_rn(a1, __fmul2_rn(sx2, make_float2(cs.z, cs.w)), make_float2(cb.z, cb.w));
    o[2 * j] = Num<OutT>::pack2(y0.x, y0.y);
    o[2 * j + 1] = Num<OutT>::pack2(y1.x, y1.y);
  }
  if (acc_dbg != nullptr && row < M) {
    int32_t* arow = acc_dbg + static_cast<size_t>(row) * N + n0 + c;
#pragma unroll
    for (int j = 0; j < 32; ++j)
      if (n0 + c + j < N) arow[j] = __float2int_rn(__uint_as_float(r[j]));
  }
  if (mapY != nullptr) {
    uint8_t* sb = staging + (NBUF > 1 ? (store_count & 1) * EPI_BYTES : 0);
    // The store that last used sb has finished reading it.
    if (lane == 0) bulk_wait_read<NBUF - 1>();
    __syncwarp();
    uint8_t* srow = sb + lane * 64;
    const int sw = (lane >> 1) & 3;
#pragma unroll
    for (int q = 0; q < 4; ++q)
      *reinterpret_cast<uint4*>(srow + ((q ^ sw) << 4)) =
          make_uint4(o[4 * q], o[4 * q + 1], o[4 * q + 2], o[4 * q + 3]);
    fence_proxy_async_smem();
    __syncwarp();
    if (lane == 0) {
      tma_store_2d(mapY, sb, n0 + c, m0 + quarter * 32);
      bulk_commit();
    }
    ++store_count;
  } else if (row < M) {
    uint16_t* yrow = static_cast<uint16_t*>(Y) + static_cast<size_t>(row) * N + n0 + c;
#pragma unroll
    for (int j = 0; j < 16; ++j) {
      if (n0 + c + 2 * j < N) yrow[2 * j] = static_cast<uint16_t>(o[j] & 0xFFFFu);
      if (n0 + c + 2 * j + 1 < N) yrow[2 * j + 1] = static_cast<uint16_t>(o[j] >> 16);
    }
  }
}

// One warp's share of a tile's epilogue: TMEM lanes 32 * quarter .. + 31
// (the warp's rows) and tile columns [col0, col0 + NCOL).  With PREFETCH the
// TMEM load of the next 32 columns is issued before the current block is
// processed, so its latency hides behind the arithmetic and the store (32
// more registers a thread).  `store_count` counts this warp's stores (it
// selects the staging buffer).
//
// SEP3 > 0: the accumulator is the sum of three TMEM accumulators SEP3
// columns apart, each an exact integer in fp32 (the W8A8 plane products); they
// are added as int32 and the block goes on with that (exact) sum.
template <typename OutT, int NCOL, int NBUF, bool PREFETCH, bool ASYM = false, int SEP3 = 0>
__device__ __forceinline__ void epilogue_part(uint32_t tmem_acc, int quarter, int col0,
                                              int lane, int m0, int n0, int M, int N, float sx,
                                              const float* col_scale, const float* col_bias,
                                              float zm, const float* col_zw,
                                              uint8_t* staging, const CUtensorMap* mapY,
                                              void* Y, int32_t* acc_dbg, int& store_count) {
  static_assert(NCOL % EPI_COLS == 0, "column share must be whole 32-column blocks");
  const uint32_t lane_base = tmem_acc + (static_cast<uint32_t>(quarter * 32) << 16);
  if (n0 + col0 >= N) return;
  if constexpr (SEP3 > 0) {
    const int row = m0 + quarter * 32 + lane;
#pragma unroll 1
    for (int c = col0; c < col0 + NCOL && n0 + c < N; c += EPI_COLS) {
      uint32_t r[32], r1[32];
      tmem_ld32(lane_base + c, r);
      tmem_ld32(lane_base + SEP3 + c, r1);
      tmem_ld_wait_tie(r);
      tmem_ld_wait_tie(r1);
      int32_t isum[32];
#pragma unroll
      for (int j = 0; j < 32; ++j)
        isum[j] = __float2int_rn(__uint_as_float(r[j])) + __float2int_rn(__uint_as_float(r1[j]));
      tmem_ld32(lane_base + 2 * SEP3 + c, r1);
      tmem_ld_wait_tie(r1);
#pragma unroll
      for (int j = 0; j < 32; ++j) {
        isum[j] += __float2int_rn(__uint_as_float(r1[j]));
        r[j] = __float_as_uint(static_cast<float>(isum[j]));
      }
      if (acc_dbg != nullptr && row < M) {
        int32_t* arow = acc_dbg + static_cast<size_t>(row) * N + n0 + c;
#pragma unroll
        for (int j = 0; j < 32; ++j)
          if (n0 + c + j < N) arow[j] = isum[j];
      }
      epilogue_block<OutT, NBUF, ASYM>(r, c, quarter, lane, m0, n0, M, N, sx, col_scale,
                                       col_bias, zm, col_zw, staging, mapY, Y, nullptr,
                                       store_count);
    }
    return;
  }
  if (!PREFETCH) {
#pragma unroll 1
    for (int c = col0; c < col0 + NCOL && n0 + c < N; c += EPI_COLS) {
      uint32_t r[32];
      tmem_ld32(lane_base + c, r);
      tmem_ld_wait_tie(r);
      epilogue_block<OutT, NBUF, ASYM>(r, c, quarter, lane, m0, n0, M, N, sx, col_scale,
                                       col_bias, zm, col_zw, staging, mapY, Y, acc_dbg,
                                       store_count);
    }
    return;
  }
  uint32_t ra[32], rb[32];
  tmem_ld32(lane_base + col0, ra);
#pragma unroll 1
  for (int c = col0; c < col0 + NCOL; c += 2 * EPI_COLS) {
    // ra holds block c (issued earlier); warp-uniform conditions throughout.
    tmem_ld_wait_tie(ra);
    const bool more1 = c + EPI_COLS < col0 + NCOL && n0 + c + EPI_COLS < N;
    if (more1) tmem_ld32(lane_base + c + EPI_COLS, rb);
    epilogue_block<OutT, NBUF, ASYM>(ra, c, quarter, lane, m0, n0, M, N, sx, col_scale,
                                     col_bias, zm, col_zw, staging, mapY, Y, acc_dbg,
                                     store_count);
    if (!more1) break;
    tmem_ld_wait_tie(rb);
    const bool more2 = c + 2 * EPI_COLS < col0 + NCOL && n0 + c + 2 * EPI_COLS < N;
    if (more2) tmem_ld32(lane_base + c + 2 * EPI_COLS, ra);
    epilogue_block<OutT, NBUF, ASYM>(rb, c + EPI_COLS, quarter, lane, m0, n0, M, N, sx,
                                     col_scale, col_bias, zm, col_zw, staging, mapY, Y,
                                     acc_dbg, store_count);
    if (!more2) break;
  }
}

}  // namespace gemm
}  // namespace clq
