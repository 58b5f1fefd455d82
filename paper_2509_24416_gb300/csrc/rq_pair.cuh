// Paired-row rotate-quantize: the hot-path variant of the tile loop in
// rq_device.cuh, for symmetric 4-bit activation codes (b >= 16, no clip):
// the OBS transform of arxiv 2509.24416 Sec. 3.3 (column gather by the swap
// vector, block Sylvester Hadamard H_b) followed by per-token symmetric
// quantization with a dynamic fp32 scale (Sec. 3.1, Eq. 1 with l = -r).
//
// What differs from the general loop: every thread works on TWO rows at the
// same permuted positions.  A tile of 2 RH rows is copied as two halves, rows
// [0, RH) to the start of the stage and rows [RH, 2 RH) HALF bytes further
// (HALF a compile-time constant), so one set of 32 gather addresses per
// thread serves both rows, the second with an immediate offset.  The tile's
// fixed costs (barrier wait, CTA barrier, scale arithmetic, loop control) are
// shared by 64 elements a thread instead of 32, and the two rows' dependency
// chains interleave.  Tiles are dealt round-robin over the grid (no claim
// counter), each CTA keeps STAGES tiles in flight, and the row maxima use
// three-input max instructions.  While the previous kernel drains, the CTA
// sets up its barriers, prefetches its first tiles into L2 and builds its
// gather addresses from the swap vector (a layer constant); X is read only
// after the programmatic-launch wait.
//
// Per tile, per thread (row r of each half, segment seg of 32 positions):
//  1. gather both rows' 32 elements from the raw stage at columns
//     perm[32 seg + (k ^ m)] (m: the XOR order of rq_device.cuh, which only
//     flips signs that the store restores) with the first butterfly stage on
//     the way in;
//  2. the remaining stages (in registers up to stride 16, across lanes above),
//     |x| maxima, warp reductions, shared atomicMax per row;
//  3. one CTA barrier, then scales, codes and 16-byte (E4M3, packed) or
//     8-byte (E2M3) stores for both rows.
#pragma once

#include "rq_device.cuh"

namespace clq {
namespace rq {

// Register cap of the paired kernel: 16 warps per SM.
constexpr int kPairMaxRegs = 128;
// Stages in flight per CTA and the two half-stage sizes (a row of K 16-bit
// elements must fit one half: the small one up to K = 8192).
constexpr int kPairStages = 2;
constexpr int kPairHalfSmall = 16 * 1024;
constexpr int kPairHalfLarge = 32 * 1024;

// Shared memory of the paired loop: STAGES stages of NR HALF bytes, row
// maxima [3][2][RH], STAGES barriers, abort flag.
__host__ __device__ inline size_t pair_smem_bytes(int RH, int half, int stages, int nr = 2) {
  return static_cast<size_t>(stages) * nr * half + 24u * RH + 8u + 8u * stages + 16u;
}

// 2^64, exactly.
#define kTwo64 __int_as_float(0x5F800000)

// |x| maximum of three values.
__device__ __forceinline__ float max3_abs(float a, float b, float c) {
  float d;
  asm("max.f32 %0, %1, %2, %3;" : "=f"(d) : "f"(fabsf(a)), "f"(fabsf(b)), "f"(fabsf(c)));
  return d;
}

__device__ __forceinline__ float max3(float a, float b, float c) {
  float d;
  asm("max.f32 %0, %1, %2, %3;" : "=f"(d) : "f"(a), "f"(b), "f"(c));
  return d;
}

// max_k |v[k]| over the 32 values of a segment (a tree of three-input maxima).
__device__ __forceinline__ float seg_absmax(const float2 (&v)[16]) {
  float m[11];
#pragma unroll
  for (int i = 0; i < 10; ++i) {
    const int e = 3 * i;  // elements e, e + 1, e + 2 of the 32
    const float x0 = (e & 1) ? v[e >> 1].y : v[e >> 1].x;
    const float x1 = ((e + 1) & 1) ? v[(e + 1) >> 1].y : v[(e + 1) >> 1].x;
    const float x2 = ((e + 2) & 1) ? v[(e + 2) >> 1].y : v[(e + 2) >> 1].x;
    m[i] = max3_abs(x0, x1, x2);
  }
  m[10] = fmaxf(fabsf(v[15].x), fabsf(v[15].y));
  const float a = max3(m[0], m[1], m[2]), b = max3(m[3], m[4], m[5]);
  const float c = max3(m[6], m[7], m[8]);
  return max3(max3(a, b, c), m[9], m[10]);
}

// Butterfly stages of one row's segment: strides 2 .. min(b, 32) / 2 in
// registers (v[k] holds positions 2k, 2k + 1, stride 1 already done), then
// strides 32 .. b / 2 across lanes.
template <int LOGB>
__device__ __forceinline__ void seg_butterflies(float2 (&v)[16], int lane) {
  const float2 neg1 = make_float2(-1.f, -1.f);
#pragma unroll
  for (int hp = 1; hp < 16; hp <<= 1) {
    if (2 * hp < (1 << LOGB)) {
#pragma unroll
      for (int k = 0; k < 16; ++k) {
        if ((k & hp) == 0) {
          const float2 x0 = v[k], x1 = v[k + hp];
          v[k] = __fadd2_rn(x0, x1);
          v[k + hp] = __ffma2_rn(x1, neg1, x0);
        }
      }
    }
  }
#pragma unroll
  for (int hl = 1; hl < 8; hl <<= 1) {
    if (LOGB > 5 && hl < (1 << (LOGB > 5 ? LOGB - 5 : 0))) {
      const float sg = (lane & hl) ? -1.f : 1.f;
      const float2 sg2 = make_float2(sg, sg);
#pragma unroll
      for (int k = 0; k < 16; ++k) {
        float2 p;
        p.x = __shfl_xor_sync(0xffffffffu, v[k].x, hl);
        p.y = __shfl_xor_sync(0xffffffffu, v[k].y, hl);
        v[k] = __ffma2_rn(v[k], sg2, p);  // lower lane: x + p, upper lane: p - x
      }
    }
  }
}

// Scale, codes and stores of one row's segment; `am` is the row's |x| maximum.
template <int CODES, bool ROT>
__device__ __forceinline__ void seg_quant_store(const RotateQuantArgs& a, float2 (&v)[16],
                                                int row, int seg, float am,
                                                uint32_t flip_words) {
  const int K = a.K;
  // s = am / 7 by division by a constant known in advance (Brisebarre,
  // Muller and Raina, IEEE Trans. Computers 53(8), 2004), as in rq_device.cuh
  constexpr float rdiv = 1.0f / 7.0f;
  const float q1 = am * rdiv;
  const float s_row = fmaf(fmaf(-7.0f, q1, am), rdiv, q1);
  if (seg == 0) a.S[row] = s_row;
  if (ROT) {
    float4* dst = reinterpret_cast<float4*>(a.rot + static_cast<size_t>(row) * K + seg * 32);
#pragma unroll
    for (int q = 0; q < 8; ++q) {
      const float sg = ((flip_words >> q) & 1u) ? -1.f : 1.f;
      dst[q] = make_float4(sg * v[2 * q].x, sg * v[2 * q].y, sg * v[2 * q + 1].x,
                           sg * v[2 * q + 1].y);
    }
  }
  // v <- rint(v / s) + 1.5 * 2^23 (ties to even), v / s as v * rcp(s); a zero
  // row gets zero codes.  A subnormal s (row maximum below about 8e-38) has no
  // approximate reciprocal: v and s are both scaled by 2^64 first (exact,
  // v <= 7 s stays far from overflow), which leaves v / s unchanged.
  const float2 magic = make_float2(12582912.0f, 12582912.0f);
  float s_div = s_row;
  if (s_row > 0.f && s_row < 1.17549435e-38f) {
    s_div = s_row * kTwo64;  // 2^64
#pragma unroll
    for (int k = 0; k < 16; ++k) v[k] = __fmul2_rn(v[k], make_float2(kTwo64, kTwo64));
  }
  const float rcp = s_div > 0.f ? rcp_approx(s_div) : 0.f;
  const float2 rc2 = make_float2(rcp, rcp);
#pragma unroll
  for (int k = 0; k < 16; ++k) v[k] = __ffma2_rn(v[k], rc2, magic);
  const float2 nmagic = make_float2(-12582912.0f, -12582912.0f);
  if constexpr (CODES == 1) {
    // one E4M3 byte a code; XOR-order signs restored on the sign bits
    uint32_t w[8];
#pragma unroll
    for (int k = 0; k < 16; k += 2) {
      uint32_t h[2];
#pragma unroll
      for (int j = 0; j < 2; ++j) {
        const float2 q = __fadd2_rn(v[k + j], nmagic);
        uint16_t e;
        asm("cvt.rn.satfinite.e4m3x2.f32 %0, %1, %2;" : "=h"(e) : "f"(q.y), "f"(q.x));
        h[j] = e;
      }
      w[k >> 1] = (h[0] | (h[1] << 16)) ^ ((0u - ((flip_words >> (k >> 1)) & 1u)) & 0x80808080u);
    }
    uint4* qrow = reinterpret_cast<uint4*>(a.Q + static_cast<size_t>(row) * K + seg * 32);
    qrow[0] = make_uint4(w[0], w[1], w[2], w[3]);
    qrow[1] = make_uint4(w[4], w[5], w[6], w[7]);
  } else if constexpr (CODES == 3) {
    // E2M3, 16 codes in 12 bytes (the packing of rq_device.cuh)
    uint32_t g[8];
#pragma unroll
    for (int k = 0; k < 16; k += 2) {
      uint32_t h[2];
#pragma unroll
      for (int j = 0; j < 2; ++j) {
        const float2 q = __fadd2_rn(v[k + j], nmagic);
        uint16_t e;
        asm("cvt.rn.satfinite.e2m3x2.f32 %0, %1, %2;" : "=h"(e) : "f"(q.y), "f"(q.x));
        h[j] = e;
      }
      uint32_t c = h[0] | (h[1] << 16);
      c ^= (0u - ((flip_words >> (k >> 1)) & 1u)) & 0x20202020u;
      const uint32_t t = c - 3u * ((c >> 2) & 0x0FC00FC0u);
      g[k >> 1] = t - 15u * ((t >> 4) & 0x00FFF000u);
    }
    uint2* qrow =
        reinterpret_cast<uint2*>(a.Q + static_cast<size_t>(row) * (3 * K / 4) + seg * 24);
    qrow[0] = make_uint2(g[0] | (g[1] << 24), (g[1] >> 8) | (g[2] << 16));
    qrow[1] = make_uint2((g[2] >> 16) | (g[3] << 8), g[4] | (g[5] << 24));
    qrow[2] = make_uint2((g[5] >> 8) | (g[6] << 16), (g[6] >> 16) | (g[7] << 8));
  } else {
    // packed nibbles: the low four bits of v are the code's two's complement
    // (no XOR order on this path: flip_words is 0)
    uint32_t by[16];
#pragma unroll
    for (int k = 0; k < 16; ++k)
      by[k] = (__float_as_uint(v[k].x) & 0xFu) | ((__float_as_uint(v[k].y) << 4) & 0xF0u);
    uint32_t w[4];
#pragma unroll
    for (int q = 0; q < 4; ++q)
      w[q] = prmt_b32(prmt_b32(by[4 * q], by[4 * q + 1], 0x0040u),
                      prmt_b32(by[4 * q + 2], by[4 * q + 3], 0x0040u), 0x5410u);
    *reinterpret_cast<uint4*>(a.Q + static_cast<size_t>(row) * (K >> 1) + seg * 16) =
        make_uint4(w[0], w[1], w[2], w[3]);
  }
}

// Bounded wait for a phase of `bar` (the rules of mbar_wait_bounded), inline
// so that no call forces the loop's registers out around it.
__device__ __forceinline__ bool pair_wait(uint64_t* bar, uint32_t parity, volatile int32_t* abort,
                                          int32_t* status) {
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = global_timer_ns();
  while (true) {
#pragma unroll 1
    for (int i = 0; i < 8; ++i)
      if (mbar_try_wait(bar, parity)) return true;
    if (*abort != 0) return false;
    if (global_timer_ns() - t0 > kWaitLimitNs) {
      record_status(status, CLQ_ERR_TIMEOUT);
      *abort = 1;
      return false;
    }
  }
}

// Copies of tile t (rows [NR RH t, NR RH t + NR RH)) into stage `dst`: the
// first RH rows at dst, the next RH (NR = 2) at dst + HALF.
template <int HALF, int NR>
__device__ __forceinline__ void pair_issue(const RotateQuantArgs& a, uint8_t* dst, uint64_t* bar,
                                           int RH, int t) {
  const int row0 = NR * RH * t;
  const int nA = max(0, min(RH, a.M - row0));
  const int nB = NR == 2 ? max(0, min(RH, a.M - row0 - RH)) : 0;
  const uint32_t row_bytes = static_cast<uint32_t>(a.K) * 2u;
  mbar_arrive_expect_tx(bar, row_bytes * static_cast<uint32_t>(nA + nB));
  const char* x = static_cast<const char*>(a.X);
  const size_t ldb = static_cast<size_t>(a.ld) * 2u;
  if (a.ld == a.K) {
    bulk_load(dst, x + static_cast<size_t>(row0) * ldb, row_bytes * nA, bar);
    if (nB > 0)
      bulk_load(dst + HALF, x + static_cast<size_t>(row0 + RH) * ldb, row_bytes * nB, bar);
  } else {
    for (int r = 0; r < nA; ++r)
      bulk_load(dst + r * row_bytes, x + static_cast<size_t>(row0 + r) * ldb, row_bytes, bar);
    for (int r = 0; r < nB; ++r)
      bulk_load(dst + HALF + r * row_bytes, x + static_cast<size_t>(row0 + RH + r) * ldb,
                row_bytes, bar);
  }
}

// L2 prefetch of the rows pair_issue(.., t) copies (ld == K: one range).
template <int NR>
__device__ __forceinline__ void pair_prefetch(const RotateQuantArgs& a, int RH, int t) {
  const int row0 = NR * RH * t;
  const int n = max(0, min(NR * RH, a.M - row0));
  const size_t row_bytes = static_cast<size_t>(a.K) * 2u;
  if (a.ld == a.K && n > 0)
    bulk_prefetch_l2(static_cast<const char*>(a.X) + static_cast<size_t>(row0) * row_bytes,
                     static_cast<uint32_t>(row_bytes * n));
}

// CODES: 0 packed nibbles, 1 E4M3, 3 E2M3.  ROT: also write the rotated rows
// to a.rot (a test aid; the variant without it keeps every value in
// registers).  NR: rows a thread works on (2: the paired loop; 1: one row, a
// stage of HALF bytes, fewer registers and so more warps per SM).
// a.rows_per_tile = RH, the rows of one half (RH K 2 bytes <= HALF,
// RH * K / 32 <= blockDim.x).
template <int NR>
constexpr int pair_max_regs() {
  return NR == 2 ? kPairMaxRegs : 96;
}

template <typename T, int LOGB, int CODES, int HALF, int STAGES, bool ROT, int NR = 2>
__global__ void __maxnreg__(pair_max_regs<NR>()) rotate_quant_pair_kernel(RotateQuantArgs a) {
  extern __shared__ __align__(16) uint8_t smem[];
  constexpr int STRIDE = NR * HALF;
  static_assert(NR == 1 || NR == 2, "one or two rows a thread");
  static_assert(LOGB >= 4 && LOGB <= 8, "paired loop: 16 <= b <= 256");
  const int K = a.K;
  const int segs = K >> 5;
  const int RH = a.rows_per_tile;
  const int tid = threadIdx.x;
  const int lane = tid & 31;
  const uint32_t row_bytes = static_cast<uint32_t>(K) * 2u;

  uint8_t* raw = smem;
  uint32_t* amax = reinterpret_cast<uint32_t*>(smem + STAGES * STRIDE);  // [3][2][RH]
  uint64_t* full = reinterpret_cast<uint64_t*>(
      (reinterpret_cast<uintptr_t>(amax + 6 * RH) + 7) & ~static_cast<uintptr_t>(7));
  int32_t* abort = reinterpret_cast<int32_t*>(full + STAGES);

  const int ntiles = (a.M + NR * RH - 1) / (NR * RH);
  if (tid == 0) {
    for (int s = 0; s < STAGES; ++s) mbar_init(&full[s], 1);
    *abort = 0;
    fence_mbarrier_init();
  }
  for (int i = tid; i < 6 * RH; i += blockDim.x) amax[i] = 0u;
  __syncthreads();
  // This CTA's first tiles into L2 while the previous kernel drains; the
  // copies after the wait still read every value from L2 / memory, where the
  // previous kernel's writes land.
  if (tid == 0)
    for (int s = 0; s < STAGES; ++s) {
      const int t = static_cast<int>(blockIdx.x) + s * static_cast<int>(gridDim.x);
      if (t < ntiles) pair_prefetch<NR>(a, RH, t);
    }
  const int items = RH * segs;
  const bool active = tid < items;
  const int r = active ? tid / segs : 0;
  const int seg = active ? tid - r * segs : 0;
  // XOR order of the gather (see rq_device.cuh): m a multiple of 8 that
  // differs between neighbouring lane groups; not for packed codes, whose
  // sign restore would cost a negation per code.
  const bool xor_order = CODES != 0 && (reinterpret_cast<uintptr_t>(a.perm) & 15u) == 0;
  const int xm = xor_order ? ((8 * (lane >> (LOGB > 5 ? LOGB - 5 : 0))) &
                              ((1 << (LOGB < 5 ? LOGB : 5)) - 8))
                           : 0;
  uint32_t flip_words = 0;
#pragma unroll
  for (int q = 0; q < 8; ++q)
    if (__popc(q & (xm >> 2)) & 1) flip_words |= 1u << q;
  uint32_t src[32];
  {
    const uint32_t base = smem_addr(raw) + static_cast<uint32_t>(r) * row_bytes;
    const int32_t* pp = a.perm + seg * 32;
    bool bad = false;
    if ((reinterpret_cast<uintptr_t>(a.perm) & 15u) == 0) {
#pragma unroll
      for (int q = 0; q < 8; ++q) {
        const int4 t = active ? __ldg(reinterpret_cast<const int4*>(pp) + (q ^ (xm >> 2)))
                              : make_int4(0, 0, 0, 0);
        const int c4[4] = {t.x, t.y, t.z, t.w};
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const bool out = static_cast<unsigned>(c4[e]) >= static_cast<unsigned>(K);
          bad |= out;
          src[4 * q + e] = base + 2u * static_cast<uint32_t>(out ? 0 : c4[e]);
        }
      }
    } else {
#pragma unroll
      for (int k = 0; k < 32; ++k) {
        const int c = active ? __ldg(pp + k) : 0;
        const bool out = static_cast<unsigned>(c) >= static_cast<unsigned>(K);
        bad |= out;
        src[k] = base + 2u * static_cast<uint32_t>(out ? 0 : c);
      }
    }
    if (bad) record_status(a.status, CLQ_ERR_DEVICE_INDEX);
  }
  // Lanes of this warp on the same row (fixed for the launch); padding lanes
  // keep the shuffles convergent and never reach a row maximum.
  const unsigned grp = __match_any_sync(0xffffffffu, active ? r : -1);
  const int leader = __ffs(grp) - 1;
  // X is read only from here on (the swap vector above is a layer constant,
  // which no kernel of this library writes).
  pdl_wait();
  pdl_launch_dependents();
  if (tid == 0)
    for (int s = 0; s < STAGES; ++s) {
      const int t = static_cast<int>(blockIdx.x) + s * static_cast<int>(gridDim.x);
      if (t < ntiles) pair_issue<HALF, NR>(a, raw + s * STRIDE, &full[s], RH, t);
    }

  bool done = false;
  for (int j0 = 0; !done; j0 += STAGES) {
#pragma unroll
    for (int s = 0; s < STAGES; ++s) {
      const int j = j0 + s;
      const int t = static_cast<int>(blockIdx.x) + j * static_cast<int>(gridDim.x);
      if (t >= ntiles) {
        done = true;
        break;
      }
      if (!pair_wait(&full[s], (j0 / STAGES) & 1, abort, a.status)) {
        done = true;
        if (tid == 0) {
          // copies already issued must land before the CTA exits
          for (int s2 = 0; s2 < STAGES; ++s2)
            for (int ph = 0; ph < 2; ++ph)
              mbar_wait_bounded(&full[s2], ph, nullptr, nullptr, 10000000ull);
        }
        break;
      }
      const int row0 = NR * RH * t;
      const int nA = min(RH, a.M - row0);
      const int nB = NR == 2 ? min(RH, a.M - row0 - RH) : 0;
      const int par = j % 3;

      // ---- 1. gather + first butterfly stage, both rows -----------------------
      float2 va[16], vb[NR == 2 ? 16 : 1];
#pragma unroll
      for (int k = 0; k < 16; ++k) {
        const uint32_t p0 = src[2 * k] + s * STRIDE, p1 = src[2 * k + 1] + s * STRIDE;
        const uint16_t x0 = lds_u16(p0), x1 = lds_u16(p1);
        va[k] = add_sub_mixed<T>(x0, to_f32<T>(x1));
        if constexpr (NR == 2) {
          const uint16_t y0 = lds_u16(p0 + HALF), y1 = lds_u16(p1 + HALF);
          vb[k] = add_sub_mixed<T>(y0, to_f32<T>(y1));
        }
      }
      // ---- 2. remaining stages, row maxima -----------------------------------
      seg_butterflies<LOGB>(va, lane);
      if constexpr (NR == 2) seg_butterflies<LOGB>(vb, lane);
      const unsigned ka = __reduce_max_sync(grp, __float_as_uint(seg_absmax(va)));
      unsigned kb = 0;
      if constexpr (NR == 2) kb = __reduce_max_sync(grp, __float_as_uint(seg_absmax(vb)));
      if (active && lane == leader) {
        if (r < nA) atomicMax(&amax[par * 2 * RH + r], ka);
        if (NR == 2 && r < nB) atomicMax(&amax[par * 2 * RH + RH + r], kb);
      }
      __syncthreads();  // row maxima complete; stage s fully read
      if (tid == 0) {
        const int t2 = t + STAGES * static_cast<int>(gridDim.x);
        if (t2 < ntiles) pair_issue<HALF, NR>(a, raw + s * STRIDE, &full[s], RH, t2);
      }
      // ---- 3. scales, codes, stores -----------------------------------------
      if (active && r < nA)
        seg_quant_store<CODES, ROT>(a, va, row0 + r, seg, __uint_as_float(amax[par * 2 * RH + r]),
                               flip_words);
      if constexpr (NR == 2)
        if (active && r < nB)
          seg_quant_store<CODES, ROT>(a, vb, row0 + RH + r, seg,
                                      __uint_as_float(amax[par * 2 * RH + RH + r]), flip_words);
      if (tid < 2 * RH) amax[((j + 2) % 3) * 2 * RH + tid] = 0u;
    }
  }
  __syncthreads();
  if (tid == 0)
    for (int s = 0; s < STAGES; ++s) mbar_inval(&full[s]);
}

}  // namespace rq
}  // namespace clq
