// Warp-specialized tcgen05 GEMM pipeline for the INT4 activation x INT4
// weight product, shared by the standalone GEMM and the fused kernel.
//
// acc[i][n] = sum_k qx[i][k] * qw[n][k] is an exact integer: |q| <= 7, so
// every product is an integer of magnitude <= 49 and, for K <= 16384, every
// partial sum stays below 2^24.  sm_103a has no integer tcgen05 MMA, so the
// codes ride on E4M3, which holds every integer in [-7, 7] exactly, through
// tcgen05.mma kind::f8f6f4 with fp32 accumulation in tensor memory; the
// integer accumulators come out exact as long as the fp32 sums are exact
// (checked bit for bit against the int64 oracle, +-7 codes at K = 16384).
// 8-bit codes (W4A8, W8A8) arrive as two E4M3 planes, 16 h and l with
// q = 16 h + l.  W4A8 multiplies both activation planes into one
// accumulator: every partial sum stays below 2^24 for K <= 16384 (at most
// (128 + 8) * 7 per code pair), so it is exact too.  W8A8 keeps three
// accumulators (SEP below) that are each exact and are added as integers.
// E2M3 operands (F6) take the same MMA with 6-bit formats.
//
// Persistent: one CTA per SM walks 128 (M) x 256 (N) tiles in a static
// round-robin order, K step 128 codes.  Each operand arrives either as E4M3
// bytes, which TMA writes straight into the MMA operand buffer with the
// 128-byte swizzle, or as packed nibbles (APACK / BPACK), which TMA stages and
// unpack warps expand into that layout.  Warp roles:
//   warp 4       TMA producer;
//   warps 6-13   unpack (only when an operand is packed; 448 threads);
//   warp 5       one lane issues tcgen05.mma (4 x K=32 per stage) and commits
//                stage and tile completion;
//   warps 0-3    epilogue (and warps 6-9 too when no operand is packed; 320
//                threads then, so 168 registers a thread): warp w drains accumulator
//                rows 32 * (w % 4) .. + 31 (the TMEM lanes its SM sub-
//                partition may read), all 256 columns with four warps, one
//                half each with eight: TMEM -> registers -> scale, bias,
//                round -> swizzled staging -> TMA tensor store.  Two TMEM
//                accumulators let the epilogue of tile i overlap the MMAs of
//                tile i + 1.
//   other warps  idle in this phase.
// With `ready` counters (fused kernel), the producer waits until all rows of
// a tile's token block have been published before loading its A tiles.
// Every wait is bounded; on a timeout the roles drain their own copies and
// MMAs and return (status word: CLQ_ERR_TIMEOUT).
#pragma once

#include "gemm_common.cuh"
#include "clq_kernels.h"

namespace clq {
namespace gemm {

constexpr int NUM_UNPACK = 256;
constexpr int WARP_TMA = 4;
constexpr int WARP_MMA = 5;
constexpr int WARP_UNPACK0 = 6;
constexpr int MIN_THREADS = (WARP_UNPACK0 + NUM_UNPACK / 32) * 32;  // 448
constexpr int MAX_STAGES = 6;

// Tile BM x BNT (BNT = 256, or 192 for E4M3 operands where N splits better).
// PA / PB: E4M3 planes per operand, 1 for 4-bit codes, 2 for 8-bit codes
// split as q = 16 h + l (plane 0 holds 16 h, plane 1 holds l; both E4M3
// values, so the MMAs of the two planes add up to q in one accumulator).
// EW: epilogue warps (0: 4 with unpack warps, else 8); SMAX: stage cap, for
// a CTA that keeps shared memory for other work.
// SEP (8-bit x 8-bit codes, PA = PB = 2): the plane products go to three
// accumulators (16 h x 16 h, the two cross terms, l x l) of one buffer, so
// that each stays exact in fp32 (see pipeline()); 3 BNT TMEM columns.
template <bool APACK, bool BPACK, int BNT = BN, int PA = 1, int PB = 1, int EW = 0,
          int SMAX = MAX_STAGES, bool SEP = false>
struct Cfg {
  static constexpr bool UNPACK = APACK || BPACK;
  static constexpr int EPI_WARPS = EW != 0 ? EW : (UNPACK ? 4 : 8);
  static constexpr int THREADS = UNPACK ? MIN_THREADS : 320;
  static constexpr int EPI_THREADS = 32 * EPI_WARPS;
  static constexpr int EPI_NBUF = 8 / EPI_WARPS;  // staging buffers per warp
  static constexpr int EPI_NCOL = BNT * 4 / EPI_WARPS;  // columns per warp
  static constexpr int AU = PA * A_U;    // E4M3 A stage (all planes)
  static constexpr int BU = PB * BNT * BK;  // E4M3 B stage (all planes)
  static constexpr int BP = BNT * BKP;   // packed B stage
  static constexpr int STAGE = AU + BU + (APACK ? A_P : 0) + (BPACK ? BP : 0);
  static constexpr int FIXED = EPI_TOTAL + 6 * BNT * 4;
  static constexpr int S0 = (222 * 1024 - FIXED) / STAGE;
  static constexpr int S = S0 > SMAX ? SMAX : S0;  // pipeline stages
  static constexpr size_t OFF_UA = 0;                           // E4M3 operands
  static constexpr size_t OFF_UB = OFF_UA + S * AU;
  static constexpr size_t OFF_PA = OFF_UB + S * BU;             // packed staging
  static constexpr size_t OFF_PB = OFF_PA + (APACK ? S * A_P : 0);
  static constexpr size_t OFF_EPI = OFF_PB + (BPACK ? S * BP : 0);
  static constexpr size_t OFF_COL = OFF_EPI + EPI_TOTAL;        // [2][3][BNT] floats
  static constexpr size_t BYTES = OFF_COL + 6 * BNT * sizeof(float);
  static constexpr uint32_t TX = (APACK ? A_P : AU) + (BPACK ? BP : BU);
  // two accumulators of BNT columns, 2 * BNT rounded up to the power of two
  // tcgen05.alloc takes
  static constexpr uint32_t TMEM = SEP ? 512u : (2 * BNT <= 256 ? 256u : 512u);
  static constexpr int NBUF = SEP ? 1 : 2;  // accumulator buffers (tiles in flight)
  static_assert(S >= 2, "pipeline needs two stages");
  static_assert((PA == 1 || PA == 2) && (PB == 1 || PB == 2), "one or two planes");
  static_assert(!UNPACK || (PA == 1 && PB == 1), "8-bit planes come as E4M3 only");
  static_assert(EPI_WARPS == 4 || (EPI_WARPS == 8 && !UNPACK), "4 or 8 epilogue warps");
  static_assert(SMAX <= MAX_STAGES, "barrier arrays hold MAX_STAGES stages");
  static_assert(!SEP || (PA == 2 && PB == 2 && 3 * BNT <= 512), "SEP: 8-bit x 8-bit, 3 BNT <= 512");
};

struct __align__(8) Barriers {
  uint64_t tma_full[MAX_STAGES];  // operand bytes landed
  uint64_t unpacked[MAX_STAGES];  // packed operands expanded (unpack warps)
  uint64_t mma_done[MAX_STAGES];  // MMAs reading the stage completed
  uint64_t acc_full[2];
  uint64_t acc_empty[2];
  uint64_t drained;
  uint32_t tmem_slot;
  int32_t abort;
};

struct Maps {
  const CUtensorMap* A;
  const CUtensorMap* B;
  const CUtensorMap* Y;   // null: direct stores
  const CUtensorMap* A2;  // second planes (PA / PB == 2), else unused
  const CUtensorMap* B2;
};

__device__ __forceinline__ uint32_t ld_acquire_u32(const uint32_t* p) {
  uint32_t v;
  asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}

__device__ __forceinline__ void fence_proxy_async_global() {
  asm volatile("fence.proxy.async.global;" ::: "memory");
}

// Barrier init (thread 0) and TMEM allocation (warp WARP_MMA); the caller
// follows with tcgen05 fences around a CTA barrier.
template <bool APACK, bool BPACK, int BNT = BN, int PA = 1, int PB = 1, int EW = 0,
          int SMAX = MAX_STAGES, bool SEP = false>
__device__ __forceinline__ void setup(Barriers* bars) {
  using C = Cfg<APACK, BPACK, BNT, PA, PB, EW, SMAX, SEP>;
  constexpr int S = C::S;
  if (threadIdx.x == 0) {
    for (int s = 0; s < S; ++s) {
      mbar_init(&bars->tma_full[s], 1);
      mbar_init(&bars->unpacked[s], NUM_UNPACK);
      mbar_init(&bars->mma_done[s], 1);
    }
    for (int s = 0; s < 2; ++s) {
      mbar_init(&bars->acc_full[s], 1);
      mbar_init(&bars->acc_empty[s], C::EPI_THREADS);
    }
    mbar_init(&bars->drained, 1);
    bars->abort = 0;
    fence_mbarrier_init();
  }
  if ((threadIdx.x >> 5) == WARP_MMA) {
    tmem_alloc(&bars->tmem_slot, C::TMEM);
    tmem_relinquish();
  }
}

// Wait (bounded) until all rows of token block m are published.
__device__ __forceinline__ bool wait_rows_ready(const uint32_t* ready, int m, uint32_t need,
                                                volatile int32_t* abort, int32_t* status) {
  const uint64_t t0 = global_timer_ns();
  while (ld_acquire_u32(ready + m) < need) {
    if (*abort != 0) return false;
    if (global_timer_ns() - t0 > kWaitLimitNs) {
      record_status(status, CLQ_ERR_TIMEOUT);
      *abort = 1;
      return false;
    }
    __nanosleep(128);
  }
  fence_proxy_async_global();
  return true;
}

// EPI_PREFETCH: let the epilogue prefetch TMEM (taken only in the 320-thread
// configuration, where registers allow it).
// ASYM: asymmetric activation codes (zero-point epilogue, g.lo / g.wsum).
// EW / SMAX: as in Cfg (the same values as the setup() call).
// F6: both operands are E2M3 codes, 16 codes in 12 bytes in global memory;
// the tensor maps (type 16U6_ALIGN16B) pad every 12-byte group to 16 bytes on
// the way into shared memory, which is the layout tcgen05.mma kind::f8f6f4
// reads for 6-bit operands, so a stage holds the same 128 bytes per row and K
// step as with E4M3 while only 96 of them cross from L2 (the copies complete
// that many transaction bytes).
//
// SEP (W8A8): plane 0 holds 16 h and plane 1 l of each 8-bit code (q = 16 h
// + l), so q_x q_w = (16 h_x)(16 h_w) + [(16 h_x) l_w + l_x (16 h_w)] + l_x l_w.
// One fp32 accumulator would round once partial sums pass 2^24 (K > 896 at
// +-127).  Kept apart, each stays exact to K = 16384: the first sums
// multiples of 256 below 2^28 (exact up to 2^32), the second multiples of 16
// below 2^25 (exact up to 2^28), the third integers below 2^20.  The
// epilogue adds them as int32 (|q_x q_w| K <= 2^28).
template <typename OutT, bool APACK, bool BPACK, int BNT = BN, bool EPI_PREFETCH = true,
          int PA = 1, int PB = 1, bool ASYM = false, int EW = 0, int SMAX = MAX_STAGES,
          bool F6 = false, bool SEP = false>
__device__ __forceinline__ void pipeline(const Maps& maps, const GemmArgs& g, uint8_t* smem,
                                         Barriers* bars, uint32_t tmem, const uint32_t* ready) {
  using C = Cfg<APACK, BPACK, BNT, PA, PB, EW, SMAX, SEP>;
  constexpr int S = C::S;
  static_assert(!F6 || (!C::UNPACK && PA == 1 && PB == 1), "E2M3 operands come one plane each");
  constexpr uint32_t TX = F6 ? C::TX / 4 * 3 : C::TX;
  volatile int32_t* abort = &bars->abort;

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int nk = (g.K + BK - 1) / BK;
  const int tiles_n = (g.N + BNT - 1) / BNT;
  const int tiles = ((g.M + BM - 1) / BM) * tiles_n;

  if (warp == WARP_TMA) {
    if (lane == 0) {
      prefetch_tensor_map(maps.A);
      prefetch_tensor_map(maps.B);
      if (PA == 2) prefetch_tensor_map(maps.A2);
      if (PB == 2) prefetch_tensor_map(maps.B2);
      if (maps.Y != nullptr) prefetch_tensor_map(maps.Y);
      int it = 0;  // K steps issued so far (all tiles)
      int ready_m = -1;
      bool ok = true;
      for (int t = blockIdx.x; t < tiles && ok; t += gridDim.x) {
        const int mb = t / tiles_n;
        const int m0 = mb * BM;
        const int n0 = (t % tiles_n) * BNT;
        if (ready != nullptr && mb != ready_m) {
          if (!wait_rows_ready(ready, mb, static_cast<uint32_t>(min(BM, g.M - m0)), abort,
                               g.status)) {
            ok = false;
            break;
          }
          ready_m = mb;
        }
        for (int kb = 0; kb < nk; ++kb, ++it) {
          const int s = it % S;
          if (!mbar_wait_bounded(&bars->mma_done[s], ((it / S) & 1) ^ 1, abort, g.status,
                                 kWaitLimitNs)) {
            ok = false;
            break;
          }
          mbar_arrive_expect_tx(&bars->tma_full[s], TX);
          if (APACK)
            tma_load_2d(smem + C::OFF_PA + s * A_P, maps.A, kb * BKP, m0, &bars->tma_full[s]);
          else
            tma_load_2d(smem + C::OFF_UA + s * C::AU, maps.A, kb * BK, m0, &bars->tma_full[s]);
          if (PA == 2)
            tma_load_2d(smem + C::OFF_UA + s * C::AU + A_U, maps.A2, kb * BK, m0,
                        &bars->tma_full[s]);
          if (BPACK)
            tma_load_2d(smem + C::OFF_PB + s * C::BP, maps.B, kb * BKP, n0, &bars->tma_full[s]);
          else
            tma_load_2d(smem + C::OFF_UB + s * C::BU, maps.B, kb * BK, n0, &bars->tma_full[s]);
          if (PB == 2)
            tma_load_2d(smem + C::OFF_UB + s * C::BU + BNT * BK, maps.B2, kb * BK, n0,
                        &bars->tma_full[s]);
        }
      }
      // On an abort, the copies already in flight must land before exit.
      if (!ok) {
        for (int j = max(0, it - S); j < it; ++j)
          mbar_wait_bounded(&bars->tma_full[j % S], (j / S) & 1, nullptr, nullptr, 10000000ull);
      }
    }
  } else if (warp == WARP_MMA) {
    if (lane == 0) {
      constexpr uint32_t idesc = F6 ? idesc_f8f6f4_f32(BM, BNT, kFmtE2M3, kFmtE2M3)
                                    : idesc_e4m3_f32(BM, BNT);
      int it = 0, tc = 0;
      bool ok = true;
      for (int t = blockIdx.x; t < tiles && ok; t += gridDim.x, ++tc) {
        const int buf = SEP ? 0 : (tc & 1);
        const uint32_t use = SEP ? tc : (tc >> 1);  // this buffer's earlier tiles
        if (!mbar_wait_bounded(&bars->acc_empty[buf], (use & 1) ^ 1, abort, g.status,
                               kWaitLimitNs)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t d = tmem + buf * BNT;
        for (int kb = 0; kb < nk; ++kb, ++it) {
          const int s = it % S;
          uint64_t* ready_bar = C::UNPACK ? &bars->unpacked[s] : &bars->tma_full[s];
          if (!mbar_wait_bounded(ready_bar, (it / S) & 1, abort, g.status, kWaitLimitNs)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t a0 = smem_addr(smem + C::OFF_UA + s * C::AU);
          const uint32_t b0 = smem_addr(smem + C::OFF_UB + s * C::BU);
#pragma unroll
          for (int pa = 0; pa < PA; ++pa)
#pragma unroll
            for (int pb = 0; pb < PB; ++pb)
#pragma unroll
              for (int k = 0; k < BK / 32; ++k) {
                // SEP: accumulator 0 (16h x 16h), 1 (cross terms), 2 (l x l); the
                // cross terms' second product always accumulates
                const int acc_i = SEP ? (pa + pb) : 0;
                const bool first = SEP ? ((kb | k) == 0 && !(pa == 1 && pb == 0))
                                       : (kb | pa | pb | k) == 0;
                mma_e4m3(d + acc_i * BNT, sw128_desc(a0 + pa * A_U + k * 32),
                         sw128_desc(b0 + pb * BNT * BK + k * 32), idesc, first ? 0u : 1u);
              }
          mma_commit(&bars->mma_done[s]);
        }
        if (ok) mma_commit(&bars->acc_full[buf]);
      }
      // Every MMA issued must complete before TMEM is released.
      mma_commit(&bars->drained);
      mbar_wait_bounded(&bars->drained, 0, nullptr, nullptr, 10000000ull);
    }
  } else if (warp < 4 || (C::EPI_WARPS == 8 && warp >= 6 && warp < 10)) {
    // ---- epilogue ----
    const int quarter = warp & 3;
    const int part = warp < 4 ? 0 : 1;                // 0: warps 0-3, 1: warps 6-9
    const int et = part * 128 + quarter * 32 + lane;  // 0 .. EPI_THREADS - 1
    uint8_t* staging = smem + C::OFF_EPI + (part * 4 + quarter) * C::EPI_NBUF * EPI_BYTES;
    int tc = 0, stores = 0;
    for (int t = blockIdx.x; t < tiles; t += gridDim.x, ++tc) {
      const int m0 = (t / tiles_n) * BM;
      const int n0 = (t % tiles_n) * BNT;
      const int buf = SEP ? 0 : (tc & 1);
      const uint32_t use = SEP ? tc : (tc >> 1);
      // Column data of this tile into the buffer of its parity; the buffer of
      // the other parity may still be read by slower warps (previous tile).
      float* col_scale = reinterpret_cast<float*>(smem + C::OFF_COL) + buf * 3 * BNT;
      float* col_bias = col_scale + BNT;
      float* col_zw = col_scale + 2 * BNT;
      for (int j = et; j < BNT; j += C::EPI_THREADS) {
        const int col = n0 + j;
        float sc = 0.f, bi = 0.f;
        if (col < g.N) {
          sc = g.s_w[col] * g.inv_b;
          if (g.bias != nullptr) bi = Num<OutT>::to_f(static_cast<const uint16_t*>(g.bias)[col]);
        }
        col_scale[j] = sc;
        col_bias[j] = bi;
        if (ASYM) col_zw[j] = col < g.N ? g.wsum[col] * sc : 0.f;
      }
      bool ok = mbar_wait_bounded(&bars->acc_full[buf], use & 1, abort, g.status,
                                  kWaitLimitNs);
      ok = __all_sync(0xffffffffu, ok);
      named_bar_sync(kEpiBarrier, C::EPI_THREADS);  // column data of this tile written
      if (!ok || *abort != 0) break;
      tc_fence_after();
      // s_x may have been written by other CTAs of this grid (fused kernel):
      // read it from L2, after the tile's MMAs have completed.
      const int row = m0 + quarter * 32 + lane;
      const float sx = row < g.M ? __ldcg(g.s_x + row) : 0.f;
      // asymmetric codes: the value of code 0 is min + 2^(n-1) delta
      const float zm = ASYM && row < g.M ? fmaf(g.zp_shift, sx, __ldcg(g.lo + row)) : 0.f;
      epilogue_part<OutT, C::EPI_NCOL, C::EPI_NBUF, EPI_PREFETCH && !C::UNPACK && !SEP, ASYM,
                    SEP ? BNT : 0>(
          tmem + buf * BNT, quarter, part * C::EPI_NCOL, lane, m0, n0, g.M, g.N, sx, col_scale,
          col_bias, zm, col_zw, staging, maps.Y, g.Y, g.acc_dbg, stores);
      tc_fence_before();
      mbar_arrive(&bars->acc_empty[buf]);
    }
    if (lane == 0) bulk_wait_all();
  } else if (C::UNPACK && warp >= WARP_UNPACK0 && warp < WARP_UNPACK0 + NUM_UNPACK / 32) {
    const int ut = threadIdx.x - WARP_UNPACK0 * 32;
    int it = 0;
    bool ok = true;
    for (int t = blockIdx.x; t < tiles && ok; t += gridDim.x) {
      for (int kb = 0; kb < nk; ++kb, ++it) {
        const int s = it % S;
        if (!mbar_wait_bounded(&bars->tma_full[s], (it / S) & 1, abort, g.status,
                               kWaitLimitNs)) {
          ok = false;
          break;
        }
        if (APACK)
          unpack_rows<BM, NUM_UNPACK>(smem + C::OFF_PA + s * A_P, smem + C::OFF_UA + s * C::AU,
                                      ut);
        if (BPACK)
          unpack_rows<BNT, NUM_UNPACK>(smem + C::OFF_PB + s * C::BP,
                                       smem + C::OFF_UB + s * C::BU, ut);
        fence_proxy_async_smem();
        mbar_arrive(&bars->unpacked[s]);
      }
    }
  }
}

// After a CTA barrier that follows pipeline(): release TMEM.
__device__ __forceinline__ void teardown(uint32_t tmem, uint32_t cols) {
  if ((threadIdx.x >> 5) == WARP_MMA) {
    tc_fence_after();
    tmem_dealloc(tmem, cols);
  }
}

}  // namespace gemm
}  // namespace clq
