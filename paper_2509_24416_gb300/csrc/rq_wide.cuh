// Wide-segment rotate-quantize: the hot-path variant of the tile loop for
// 4-bit activation codes when b >= 64 and K % 64 == 0 (the OBS transform of
// arxiv 2509.24416 Sec. 3.3 and the per-token quantization of Sec. 3.1 /
// Eq. 1, symmetric, or asymmetric with the row's minimum and maximum, as in
// rq_device.cuh).
//
// Each thread owns 64 consecutive permuted positions of one row, so a block
// of b = 64 is transformed entirely in its registers (b = 128 / 256 keep one /
// two stages across lanes): the cross-lane shuffles, which load the shared
// memory pipe as much as the gather does, drop out (b = 64) or halve.  The
// 64 gather offsets (bytes from the stage start, below 64 KB) are kept two to
// a register, so the thread holds as many address registers as the 32-wide
// loop while doing twice the work per tile.  The rest follows rq_pair.cuh:
// round-robin tiles, STAGES stages in flight, three-input maxima, one CTA
// barrier per tile, the XOR-ordered gather whose sign flips the store undoes,
// and a prologue that runs while the previous kernel drains: barriers, an L2
// prefetch of the first tiles and the gather offsets from the swap vector (a
// layer constant), with X read only after the programmatic-launch wait.
#pragma once

#include "rq_pair.cuh"

namespace clq {
namespace rq {

constexpr int kWideMaxRegs = 168;

// Shared memory of the wide loop: STAGES stages of STAGE bytes, row maxima
// and (asymmetric codes) row minima [3][RH] each, STAGES barriers, abort flag.
__host__ __device__ inline size_t wide_smem_bytes(int RH, int stage, int stages) {
  return static_cast<size_t>(stages) * stage + 24u * RH + 8u + 8u * stages + 16u;
}

// max_k v[k] and min_k v[k] over the 64 values of a segment.
__device__ __forceinline__ void wide_minmax(const float2 (&v)[32], float& mx, float& mn) {
  float a[16], b[16];
#pragma unroll
  for (int i = 0; i < 16; ++i) {
    a[i] = max3(fmaxf(v[2 * i].x, v[2 * i].y), v[2 * i + 1].x, v[2 * i + 1].y);
    b[i] = fminf(fminf(v[2 * i].x, v[2 * i].y), fminf(v[2 * i + 1].x, v[2 * i + 1].y));
  }
#pragma unroll
  for (int w = 8; w >= 1; w >>= 1)
#pragma unroll
    for (int i = 0; i < w; ++i) {
      a[i] = fmaxf(a[i], a[i + w]);
      b[i] = fminf(b[i], b[i + w]);
    }
  mx = a[0];
  mn = b[0];
}

// max_k |v[k]| over the 64 values of a segment.
__device__ __forceinline__ float wide_absmax(const float2 (&v)[32]) {
  float m[22];
#pragma unroll
  for (int i = 0; i < 21; ++i) {
    const int e = 3 * i;  // elements e, e + 1, e + 2 of the 64
    const float x0 = (e & 1) ? v[e >> 1].y : v[e >> 1].x;
    const float x1 = ((e + 1) & 1) ? v[(e + 1) >> 1].y : v[(e + 1) >> 1].x;
    const float x2 = ((e + 2) & 1) ? v[(e + 2) >> 1].y : v[(e + 2) >> 1].x;
    m[i] = max3_abs(x0, x1, x2);
  }
  m[21] = fabsf(v[31].y);
  float n[8];
#pragma unroll
  for (int i = 0; i < 7; ++i) n[i] = max3(m[3 * i], m[3 * i + 1], m[3 * i + 2]);
  n[7] = m[21];
  return max3(max3(n[0], n[1], n[2]), max3(n[3], n[4], n[5]), fmaxf(n[6], n[7]));
}

// Butterfly stages of a 64-wide segment: strides 2 .. min(b, 64) / 2 in
// registers (v[k] holds positions 2k, 2k + 1, stride 1 done), then strides
// 64 .. b / 2 across lanes.
template <int LOGB>
__device__ __forceinline__ void wide_butterflies(float2 (&v)[32], int lane) {
  const float2 neg1 = make_float2(-1.f, -1.f);
#pragma unroll
  for (int hp = 1; hp < 32; hp <<= 1) {
    if (2 * hp < (1 << LOGB)) {
#pragma unroll
      for (int k = 0; k < 32; ++k) {
        if ((k & hp) == 0) {
          const float2 x0 = v[k], x1 = v[k + hp];
          v[k] = __fadd2_rn(x0, x1);
          v[k + hp] = __ffma2_rn(x1, neg1, x0);
        }
      }
    }
  }
#pragma unroll
  for (int hl = 1; hl < 4; hl <<= 1) {
    if (LOGB > 6 && hl < (1 << (LOGB > 6 ? LOGB - 6 : 0))) {
      const float sg = (lane & hl) ? -1.f : 1.f;
      const float2 sg2 = make_float2(sg, sg);
#pragma unroll
      for (int k = 0; k < 32; ++k) {
        float2 p;
        p.x = __shfl_xor_sync(0xffffffffu, v[k].x, hl);
        p.y = __shfl_xor_sync(0xffffffffu, v[k].y, hl);
        v[k] = __ffma2_rn(v[k], sg2, p);  // lower lane: x + p, upper lane: p - x
      }
    }
  }
}

// Scale, codes and stores of one row's 64-wide segment; `am` is the row's
// |x| maximum; bit q of `flip` flips the signs of codes 4q .. 4q + 3.
template <int CODES, bool ROT>
__device__ __forceinline__ void wide_quant_store(const RotateQuantArgs& a, float2 (&v)[32],
                                                 int row, int seg, float am, uint32_t flip) {
  const int K = a.K;
  // s = am / 7 by division by a constant known in advance (Brisebarre,
  // Muller and Raina, IEEE Trans. Computers 53(8), 2004), as in rq_device.cuh
  constexpr float rdiv = 1.0f / 7.0f;
  const float q1 = am * rdiv;
  const float s_row = fmaf(fmaf(-7.0f, q1, am), rdiv, q1);
  if (seg == 0) a.S[row] = s_row;
  if (ROT) {
    float4* dst = reinterpret_cast<float4*>(a.rot + static_cast<size_t>(row) * K + seg * 64);
#pragma unroll
    for (int q = 0; q < 16; ++q) {
      const float sg = ((flip >> q) & 1u) ? -1.f : 1.f;
      dst[q] = make_float4(sg * v[2 * q].x, sg * v[2 * q].y, sg * v[2 * q + 1].x,
                           sg * v[2 * q + 1].y);
    }
  }
  // v <- rint(v / s) + 1.5 * 2^23 (ties to even), v / s as v * rcp(s); a zero
  // row gets zero codes; a subnormal s is scaled with v by 2^64 first.
  const float2 magic = make_float2(12582912.0f, 12582912.0f);
  float s_div = s_row;
  if (s_row > 0.f && s_row < 1.17549435e-38f) {
    s_div = s_row * kTwo64;
#pragma unroll
    for (int k = 0; k < 32; ++k) v[k] = __fmul2_rn(v[k], make_float2(kTwo64, kTwo64));
  }
  const float rcp = s_div > 0.f ? rcp_approx(s_div) : 0.f;
  const float2 rc2 = make_float2(rcp, rcp);
#pragma unroll
  for (int k = 0; k < 32; ++k) v[k] = __ffma2_rn(v[k], rc2, magic);
  const float2 nmagic = make_float2(-12582912.0f, -12582912.0f);
  if constexpr (CODES == 1) {
    uint4* qrow = reinterpret_cast<uint4*>(a.Q + static_cast<size_t>(row) * K + seg * 64);
#pragma unroll
    for (int c = 0; c < 4; ++c) {  // 16 codes a store
      uint32_t w[4];
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const int k = 8 * c + 2 * j;  // v[k], v[k + 1]: codes 2k .. 2k + 3
        uint16_t e0, e1;
        const float2 q0 = __fadd2_rn(v[k], nmagic), q1v = __fadd2_rn(v[k + 1], nmagic);
        asm("cvt.rn.satfinite.e4m3x2.f32 %0, %1, %2;" : "=h"(e0) : "f"(q0.y), "f"(q0.x));
        asm("cvt.rn.satfinite.e4m3x2.f32 %0, %1, %2;" : "=h"(e1) : "f"(q1v.y), "f"(q1v.x));
        w[j] = (static_cast<uint32_t>(e0) | (static_cast<uint32_t>(e1) << 16)) ^
               ((0u - ((flip >> (k >> 1)) & 1u)) & 0x80808080u);
      }
      qrow[c] = make_uint4(w[0], w[1], w[2], w[3]);
    }
  } else {
    // E2M3: 16 codes in 12 bytes (the packing of rq_device.cuh); 64 codes are
    // 48 bytes, three 16-byte stores
    uint32_t g[16];
#pragma unroll
    for (int k = 0; k < 32; k += 2) {
      uint16_t e0, e1;
      const float2 q0 = __fadd2_rn(v[k], nmagic), q1v = __fadd2_rn(v[k + 1], nmagic);
      asm("cvt.rn.satfinite.e2m3x2.f32 %0, %1, %2;" : "=h"(e0) : "f"(q0.y), "f"(q0.x));
      asm("cvt.rn.satfinite.e2m3x2.f32 %0, %1, %2;" : "=h"(e1) : "f"(q1v.y), "f"(q1v.x));
      uint32_t c = static_cast<uint32_t>(e0) | (static_cast<uint32_t>(e1) << 16);
      c ^= (0u - ((flip >> (k >> 1)) & 1u)) & 0x20202020u;
      const uint32_t t = c - 3u * ((c >> 2) & 0x0FC00FC0u);
      g[k >> 1] = t - 15u * ((t >> 4) & 0x00FFF000u);
    }
    uint32_t o[12];
#pragma unroll
    for (int h = 0; h < 4; ++h) {  // each group of 16 codes: g[4h .. 4h + 3] -> 3 words
      o[3 * h] = g[4 * h] | (g[4 * h + 1] << 24);
      o[3 * h + 1] = (g[4 * h + 1] >> 8) | (g[4 * h + 2] << 16);
      o[3 * h + 2] = (g[4 * h + 2] >> 16) | (g[4 * h + 3] << 8);
    }
    uint4* qrow =
        reinterpret_cast<uint4*>(a.Q + static_cast<size_t>(row) * (3 * K / 4) + seg * 48);
    qrow[0] = make_uint4(o[0], o[1], o[2], o[3]);
    qrow[1] = make_uint4(o[4], o[5], o[6], o[7]);
    qrow[2] = make_uint4(o[8], o[9], o[10], o[11]);
  }
}

// Asymmetric codes of one row's 64-wide segment (Eq. 1 with the row's
// minimum and maximum as bounds, as in rq_device.cuh): delta = (max - min) /
// 15 by the same division by a constant, q = rint((v - min) / delta) stored
// centered as q - 8 in E4M3 bytes; kmax / kmin are the row's order keys of
// max and -min.  v holds the true transform (signs already restored).
template <bool ROT>
__device__ __forceinline__ void wide_quant_store_asym(const RotateQuantArgs& a, float2 (&v)[32],
                                                      int row, int seg, uint32_t kmax,
                                                      uint32_t kmin) {
  const int K = a.K;
  constexpr float div = 15.0f;
  constexpr float rdiv = 1.0f / 15.0f;
  const float row_lo = -order_key_inv(kmin);
  const float am = __fsub_rn(order_key_inv(kmax), row_lo);
  const float q1 = am * rdiv;
  const float s_row = fmaf(fmaf(-div, q1, am), rdiv, q1);
  if (seg == 0) {
    a.S[row] = s_row;
    a.lo[row] = row_lo;
  }
  if (ROT) {
    float4* dst = reinterpret_cast<float4*>(a.rot + static_cast<size_t>(row) * K + seg * 64);
#pragma unroll
    for (int q = 0; q < 16; ++q)
      dst[q] = make_float4(v[2 * q].x, v[2 * q].y, v[2 * q + 1].x, v[2 * q + 1].y);
  }
  // v <- rint((v - min) * 15 / span) + 1.5 * 2^23 - 8 (the centered code in
  // the low mantissa bits); a constant row gets q = 0; a subnormal span takes
  // exact divisions.
  const float2 mg = make_float2(12582912.0f - 8.0f, 12582912.0f - 8.0f);
  const float2 nlo = make_float2(-row_lo, -row_lo);
  // exact divisions also where rcp(span) would be subnormal (span >= 2^126,
  // bf16 inputs near their top), which rcp.approx.ftz flushes to zero
  if (am > 0.f && (am < 1.17549435e-38f || am >= 8.50705917e37f)) {
#pragma unroll
    for (int k = 0; k < 32; ++k) {
      const float2 d = __fadd2_rn(v[k], nlo);
      v[k] = __fadd2_rn(make_float2(__fmul_rn(__fdiv_rn(d.x, am), div),
                                    __fmul_rn(__fdiv_rn(d.y, am), div)),
                        mg);
    }
  } else {
    const float inv = am > 0.f ? div * rcp_approx(am) : 0.f;
    const float2 inv2 = make_float2(inv, inv);
#pragma unroll
    for (int k = 0; k < 32; ++k) v[k] = __ffma2_rn(__fadd2_rn(v[k], nlo), inv2, mg);
  }
  const float2 nmagic = make_float2(-12582912.0f, -12582912.0f);
  uint4* qrow = reinterpret_cast<uint4*>(a.Q + static_cast<size_t>(row) * K + seg * 64);
#pragma unroll
  for (int c = 0; c < 4; ++c) {  // 16 codes a store
    uint32_t w[4];
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int k = 8 * c + 2 * j;
      uint16_t e0, e1;
      const float2 q0 = __fadd2_rn(v[k], nmagic), q1v = __fadd2_rn(v[k + 1], nmagic);
      asm("cvt.rn.satfinite.e4m3x2.f32 %0, %1, %2;" : "=h"(e0) : "f"(q0.y), "f"(q0.x));
      asm("cvt.rn.satfinite.e4m3x2.f32 %0, %1, %2;" : "=h"(e1) : "f"(q1v.y), "f"(q1v.x));
      w[j] = static_cast<uint32_t>(e0) | (static_cast<uint32_t>(e1) << 16);
    }
    qrow[c] = make_uint4(w[0], w[1], w[2], w[3]);
  }
}

// CODES 1 (E4M3) or 3 (E2M3); 64 <= b <= 256 (LOGB 6 .. 8); K % 64 == 0.
// ASYM: asymmetric codes (a.lo != null), E4M3 only.
// a.rows_per_tile = RH rows a tile (RH * 2K <= STAGE, RH * K / 64 <=
// blockDim.x).
template <typename T, int LOGB, int CODES, int STAGE, int STAGES, bool ROT, bool ASYM = false>
__global__ void __maxnreg__(kWideMaxRegs) rotate_quant_wide_kernel(RotateQuantArgs a) {
  extern __shared__ __align__(16) uint8_t smem[];
  static_assert(LOGB >= 6 && LOGB <= 8, "wide loop: 64 <= b <= 256");
  static_assert(STAGE <= 65536, "gather offsets are 16-bit");
  static_assert(!ASYM || CODES == 1, "asymmetric codes in E4M3 bytes only");
  const int K = a.K;
  const int segs = K >> 6;
  const int RH = a.rows_per_tile;
  const int tid = threadIdx.x;
  const int lane = tid & 31;
  const uint32_t row_bytes = static_cast<uint32_t>(K) * 2u;

  uint8_t* raw = smem;
  uint32_t* amax = reinterpret_cast<uint32_t*>(smem + STAGES * STAGE);  // [3][RH]
  uint32_t* amin = amax + 3 * RH;                                          // [3][RH]
  uint64_t* full = reinterpret_cast<uint64_t*>(
      (reinterpret_cast<uintptr_t>(amin + 3 * RH) + 7) & ~static_cast<uintptr_t>(7));
  int32_t* abort = reinterpret_cast<int32_t*>(full + STAGES);

  const int ntiles = (a.M + RH - 1) / RH;
  if (tid == 0) {
    for (int s = 0; s < STAGES; ++s) mbar_init(&full[s], 1);
    *abort = 0;
    fence_mbarrier_init();
  }
  for (int i = tid; i < 6 * RH; i += blockDim.x) amax[i] = 0u;  // and amin
  __syncthreads();
  // This CTA's first tiles into L2 while the previous kernel drains; the
  // copies after the wait still read every value from L2 / memory, where the
  // previous kernel's writes land.
  if (tid == 0)
    for (int s = 0; s < STAGES; ++s) {
      const int t = static_cast<int>(blockIdx.x) + s * static_cast<int>(gridDim.x);
      if (t < ntiles) pair_prefetch<1>(a, RH, t);
    }
  const int items = RH * segs;
  const bool active = tid < items;
  const int r = active ? tid / segs : 0;
  const int seg = active ? tid - r * segs : 0;
  // XOR order: register pair k holds positions (2k) ^ m, (2k + 1) ^ m, m a
  // multiple of 8 below 64 that differs between neighbouring lanes (shared by
  // the lanes a cross-lane stage joins); the transform then comes out with
  // the sign (-1)^popc(i & m) on output i, constant over each 8 codes.
  const bool xor_order = (reinterpret_cast<uintptr_t>(a.perm) & 15u) == 0;
  const int xm = xor_order ? ((8 * (lane >> (LOGB - 6))) & 56) : 0;
  uint32_t flip = 0;
#pragma unroll
  for (int q = 0; q < 16; ++q)
    if (__popc((4 * q) & xm) & 1) flip |= 1u << q;
  // Gather offsets (bytes from the stage start) of positions (2k) ^ m and
  // (2k + 1) ^ m, low and high halves of ow[k].  An index outside [0, K) is
  // reported and replaced by column 0.
  uint32_t ow[32];
  {
    const uint32_t rbase = static_cast<uint32_t>(r) * row_bytes;
    const int32_t* pp = a.perm + seg * 64;
    bool bad = false;
    auto off = [&](int c) {
      const bool out = static_cast<unsigned>(c) >= static_cast<unsigned>(K);
      bad |= out;
      return rbase + 2u * static_cast<uint32_t>(out ? 0 : c);
    };
    if (xor_order) {
#pragma unroll
      for (int q = 0; q < 16; ++q) {  // positions 4q .. 4q + 3, read in the XOR order
        const int4 t = active ? __ldg(reinterpret_cast<const int4*>(pp) + (q ^ (xm >> 2)))
                              : make_int4(0, 0, 0, 0);
        ow[2 * q] = off(t.x) | (off(t.y) << 16);
        ow[2 * q + 1] = off(t.z) | (off(t.w) << 16);
      }
    } else {
#pragma unroll
      for (int k = 0; k < 32; ++k) {
        const int c0 = active ? __ldg(pp + 2 * k) : 0;
        const int c1 = active ? __ldg(pp + 2 * k + 1) : 0;
        ow[k] = off(c0) | (off(c1) << 16);
      }
    }
    if (bad) record_status(a.status, CLQ_ERR_DEVICE_INDEX);
  }
  const uint32_t sbase = smem_addr(raw);
  const unsigned grp = __match_any_sync(0xffffffffu, active ? r : -1);
  const int leader = __ffs(grp) - 1;

  // X is read only from here on (the swap vector above is a layer constant,
  // which no kernel of this library writes).
  pdl_wait();
  pdl_launch_dependents();
  if (tid == 0)
    for (int s = 0; s < STAGES; ++s) {
      const int t = static_cast<int>(blockIdx.x) + s * static_cast<int>(gridDim.x);
      if (t < ntiles) pair_issue<STAGE, 1>(a, raw + s * STAGE, &full[s], RH, t);
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
          for (int s2 = 0; s2 < STAGES; ++s2)
            for (int ph = 0; ph < 2; ++ph)
              mbar_wait_bounded(&full[s2], ph, nullptr, nullptr, 10000000ull);
        }
        break;
      }
      const int row0 = RH * t;
      const int n = min(RH, a.M - row0);
      const int par = j % 3;

      // ---- 1. gather + first butterfly stage ------------------------------------
      float2 v[32];
      const uint32_t st = sbase + s * STAGE;
#pragma unroll
      for (int k = 0; k < 32; ++k) {
        const uint16_t x0 = lds_u16(st + (ow[k] & 0xFFFFu));
        const uint16_t x1 = lds_u16(st + (ow[k] >> 16));
        v[k] = add_sub_mixed<T>(x0, to_f32<T>(x1));
      }
      // ---- 2. remaining stages, row maximum -----------------------------------
      wide_butterflies<LOGB>(v, lane);
      if constexpr (ASYM) {
        // the bounds are signed: restore each 4-code group's sign first
        if (xor_order) {
#pragma unroll
          for (int q = 0; q < 16; ++q) {
            const float sg = ((flip >> q) & 1u) ? -1.f : 1.f;
            const float2 sg2 = make_float2(sg, sg);
            v[2 * q] = __fmul2_rn(v[2 * q], sg2);
            v[2 * q + 1] = __fmul2_rn(v[2 * q + 1], sg2);
          }
        }
        float mx, mn;
        wide_minmax(v, mx, mn);
        const unsigned kx = __reduce_max_sync(grp, order_key(mx));
        const unsigned kn = __reduce_max_sync(grp, order_key(-mn));
        if (active && lane == leader && r < n) {
          atomicMax(&amax[par * RH + r], kx);
          atomicMax(&amin[par * RH + r], kn);
        }
      } else {
        const unsigned kx = __reduce_max_sync(grp, __float_as_uint(wide_absmax(v)));
        if (active && lane == leader && r < n) atomicMax(&amax[par * RH + r], kx);
      }
      __syncthreads();  // row maxima complete; stage s fully read
      if (tid == 0) {
        const int t2 = t + STAGES * static_cast<int>(gridDim.x);
        if (t2 < ntiles) pair_issue<STAGE, 1>(a, raw + s * STAGE, &full[s], RH, t2);
      }
      // ---- 3. scale, codes, stores --------------------------------------------
      if (active && r < n) {
        if constexpr (ASYM)
          wide_quant_store_asym<ROT>(a, v, row0 + r, seg, amax[par * RH + r],
                                     amin[par * RH + r]);
        else
          wide_quant_store<CODES, ROT>(a, v, row0 + r, seg,
                                       __uint_as_float(amax[par * RH + r]), flip);
      }
      if (tid < RH) {
        amax[((j + 2) % 3) * RH + tid] = 0u;
        if (ASYM) amin[((j + 2) % 3) * RH + tid] = 0u;
      }
    }
  }
  __syncthreads();
  if (tid == 0)
    for (int s = 0; s < STAGES; ++s) mbar_inval(&full[s]);
}

}  // namespace rq
}  // namespace clq
