// Rotate-quantize tile loop, shared by the standalone kernel and the fused
// linear kernel.  It applies the OBS transform of arxiv 2509.24416 Sec. 3.3
// to rows of X (column gather by the swap vector `perm`, then the block
// Sylvester Hadamard H_b) and quantizes each row to symmetric INT4 with a
// dynamic fp32 scale (Sec. 3.1, Eq. 1 with l = -r).
//
// Every thread of the CTA takes part.  The CTA walks tiles of R rows
// (tile = blockIdx.x + i * gridDim.x).  Raw rows stream into a ring of
// `stages` shared-memory buffers with bulk asynchronous copies
// (cp.async.bulk + mbarrier), so several tiles are in flight per SM while the
// threads work on an earlier one.  Per tile:
//  phase 1: every element of the raw rows is stored to its permuted position
//           in a row buffer (scatter through the inverse of perm, built once
//           per CTA as shared-memory byte offsets);
//  phase 2: one thread per (row, 32 consecutive permuted positions) reads its
//           segment (4 x 16 B, conflict-free thanks to a chunk swizzle), runs
//           the first log2(min(b, 32)) butterfly stages in registers (paired
//           fp32x2 arithmetic) and the remaining log2(b / 32) across lanes
//           with shuffles, and reduces |x| per row;
//  phase 3: s = absmax / 7, codes rint(x * (1 / s)) via the 1.5 * 2^23
//           rounding constant (ties to even), then either packed nibbles
//           (the code's two's complement is the low nibble of the sum's bits;
//           one 16-byte store per thread) or one E4M3 byte per code (cvt of
//           the integer-valued float; two 16-byte stores per thread).
#pragma once

#include "clq_device.cuh"
#include "clq_kernels.h"

namespace clq {
namespace rq {

constexpr int kMaxStages = 4;

// Byte offset of permuted position j inside a row buffer.  16-byte chunk q
// is stored at q ^ ((q >> 3) & 3): a thread reading chunks 4s..4s+3 and its
// neighbours reading theirs hit distinct banks within every 8-lane phase.
__device__ __forceinline__ uint32_t rowbuf_offset(uint32_t j) {
  const uint32_t q = j >> 3;
  const uint32_t phys = q ^ ((q >> 3) & 3u);
  return (phys << 4) | ((j & 7u) << 1);
}

// Two packed 16-bit values (low half first) -> float2, exactly.
template <typename T>
__device__ __forceinline__ float2 to_f2(uint32_t w);
template <>
__device__ __forceinline__ float2 to_f2<__half>(uint32_t w) {
  return __half22float2(*reinterpret_cast<const __half2*>(&w));
}
template <>
__device__ __forceinline__ float2 to_f2<__nv_bfloat16>(uint32_t w) {
  return make_float2(__uint_as_float(w << 16), __uint_as_float(w & 0xFFFF0000u));
}

__device__ __forceinline__ uint32_t prmt_b32(uint32_t a, uint32_t b, uint32_t c) {
  uint32_t d;
  asm("prmt.b32 %0, %1, %2, %3;" : "=r"(d) : "r"(a), "r"(b), "r"(c));
  return d;
}

__device__ __forceinline__ void mbar_inval(uint64_t* bar) {
  asm volatile("mbarrier.inval.shared::cta.b64 [%0];" ::"r"(smem_addr(bar)) : "memory");
}

// Shared memory of the tile loop: K offsets, R row buffer rows, `stages` raw
// tiles, 2R maxima, `stages` barriers, abort flag.
__host__ __device__ inline size_t smem_bytes(int K, int R, int stages) {
  return static_cast<size_t>(4 * K) + static_cast<size_t>(R) * 2 * K * (1 + stages) + 8u * R +
         8u * kMaxStages + 16u + 4u * kMaxStages;
}

struct NoPublish {
  __device__ void operator()(int, int) const {}
};

struct Shared {
  uint32_t* off;    // [K] byte offset of column c in a row buffer
  uint8_t* rowbuf;  // [R][2K] permuted rows
  uint8_t* raw;     // [stages][R][2K] raw rows
  uint32_t* amax;   // [2][R]
  uint64_t* full;   // [stages]
  int32_t* abort;
  int32_t* tile_of; // [stages] tile held by each raw stage, -1 = none left
};

// Issue the bulk copies of tile `tile` into raw stage `s`.
__device__ __forceinline__ void issue_tile(const RotateQuantArgs& a, const Shared& sh, int R,
                                           int tile, int s) {
  const int row0 = tile * R;
  const int rows = min(R, a.M - row0);
  const uint32_t row_bytes = static_cast<uint32_t>(a.K) * 2u;
  uint8_t* dst = sh.raw + static_cast<size_t>(s) * R * row_bytes;
  const char* src = static_cast<const char*>(a.X) + static_cast<size_t>(row0) * a.ld * 2u;
  mbar_arrive_expect_tx(&sh.full[s], row_bytes * rows);
  if (a.ld == a.K) {
    bulk_load(dst, src, row_bytes * rows, &sh.full[s]);
  } else {
    for (int r = 0; r < rows; ++r)
      bulk_load(dst + static_cast<size_t>(r) * row_bytes,
                src + static_cast<size_t>(r) * a.ld * 2u, row_bytes, &sh.full[s]);
  }
}

// Runs the tile loop with every thread of the CTA.  Tiles come in a static
// round-robin order (tile_counter == null) or are claimed one at a time from
// a global counter (so that CTAs which never become resident own no rows).
// After each tile, every thread calls publish(row0, rows) once its own stores
// of that tile are issued.  LOGB = log2(b) when known at compile time, or -1
// to read a.logb.
template <typename T, int LOGB, bool CLIP, typename Publish>
__device__ __forceinline__ void run(const RotateQuantArgs& a, uint8_t* smem, int stages,
                                    uint32_t* tile_counter, Publish publish) {
  const int K = a.K;
  const int segs = K >> 5;
  const int R = a.rows_per_tile;
  const int lb = LOGB >= 0 ? LOGB : a.logb;  // log2(b): compile time or runtime
  const int nthr = blockDim.x;
  const int tid = threadIdx.x;
  const int lane = tid & 31;
  const size_t row_bytes = static_cast<size_t>(K) * 2u;

  Shared sh;
  sh.off = reinterpret_cast<uint32_t*>(smem);
  sh.rowbuf = smem + 4 * K;
  sh.raw = sh.rowbuf + R * row_bytes;
  sh.amax = reinterpret_cast<uint32_t*>(sh.raw + static_cast<size_t>(stages) * R * row_bytes);
  sh.full = reinterpret_cast<uint64_t*>(
      (reinterpret_cast<uintptr_t>(sh.amax + 2 * R) + 7) & ~static_cast<uintptr_t>(7));
  sh.abort = reinterpret_cast<int32_t*>(sh.full + kMaxStages);
  sh.tile_of = sh.abort + 4;

  const int ntiles = (a.M + R - 1) / R;
  int claims = 0;  // tid 0: tiles claimed so far
  // tid 0: claim the next tile into stage s and start its copies (or mark
  // the stage empty and complete its phase without data).
  auto refill = [&](int s) {
    int t;
    if (tile_counter != nullptr)
      t = static_cast<int>(atomicAdd(tile_counter, 1u));
    else
      t = static_cast<int>(blockIdx.x) + claims * static_cast<int>(gridDim.x);
    ++claims;
    if (t < ntiles) {
      sh.tile_of[s] = t;
      issue_tile(a, sh, R, t, s);
    } else {
      sh.tile_of[s] = -1;
      mbar_arrive(&sh.full[s]);
    }
  };

  if (tid == 0) {
    for (int s = 0; s < stages; ++s) mbar_init(&sh.full[s], 1);
    *sh.abort = 0;
    fence_mbarrier_init();
  }
  // Inverse of perm as destination offsets.  Entries default to 0 so that a
  // perm that is not a permutation produces wrong values, never a stray
  // shared-memory write; out-of-range indices are reported and skipped.
  for (int c = tid; c < K; c += nthr) sh.off[c] = 0u;
  for (int i = tid; i < 2 * R; i += nthr) sh.amax[i] = 0u;
  __syncthreads();
  if (tid == 0)
    for (int s = 0; s < stages; ++s) refill(s);
  for (int j = tid; j < K; j += nthr) {
    const int c = __ldg(a.perm + j);
    if (static_cast<unsigned>(c) < static_cast<unsigned>(K))
      sh.off[c] = rowbuf_offset(j);
    else
      record_status(a.status, CLQ_ERR_DEVICE_INDEX);
  }
  __syncthreads();

  const int items = R * segs;
  const bool active = tid < items;
  const int r_local = active ? tid / segs : 0;
  const int seg = active ? tid - r_local * segs : 0;
  const int cpr = K >> 3;  // 16-byte chunks per row
  const int pairs = R * cpr;
  bool aborted = false;

  // Phase-1 work of this thread is the same for every tile: at most four
  // (row, 16-byte chunk) pairs p = tid + u * blockDim.x (R * K / 8 <= 4 *
  // blockDim.x).  Pair p reads bytes [16p, 16p + 16) of a raw stage (rows of
  // 2K bytes are contiguous) and is live when p < rows * K / 8.  The shared
  // address of each of its 8 elements' permuted positions is computed once.
  const uint32_t rowbuf_base = smem_addr(sh.rowbuf);
  const uint32_t raw_base = smem_addr(sh.raw);
  uint32_t dst[4][8];
#pragma unroll
  for (int u = 0; u < 4; ++u) {
    const int p = tid + u * nthr;
    const int r = p < pairs ? p / cpr : 0;
    const int c = p < pairs ? p - r * cpr : 0;
#pragma unroll
    for (int e = 0; e < 8; ++e)
      dst[u][e] = rowbuf_base + static_cast<uint32_t>(r * row_bytes) + sh.off[c * 8 + e];
  }
  // Phase-2 addresses of this thread's four 16-byte chunks.
  uint32_t seg_addr[4];
#pragma unroll
  for (int c = 0; c < 4; ++c) {
    const uint32_t q = static_cast<uint32_t>(seg * 4 + c);
    seg_addr[c] = rowbuf_base + static_cast<uint32_t>(r_local * row_bytes) +
                  ((q ^ ((q >> 3) & 3u)) << 4);
  }

  for (int i = 0;; ++i) {
    const int s = i % stages;
    const int par = i & 1;
    if (!mbar_wait_bounded(&sh.full[s], (i / stages) & 1, sh.abort, a.status, kWaitLimitNs)) {
      aborted = true;
      break;
    }
    const int tile = *reinterpret_cast<volatile int32_t*>(&sh.tile_of[s]);
    if (tile < 0) break;
    const int row0 = tile * R;
    const int rows = min(R, a.M - row0);

    // ---- phase 1: raw rows -> permuted row buffer --------------------------
    const uint32_t stage_base = raw_base + static_cast<uint32_t>(s * R * row_bytes);
    const int live = rows * cpr;
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const int p = tid + u * nthr;
      if (p < live) {
        uint4 v;
        asm volatile("ld.shared.v4.u32 {%0,%1,%2,%3}, [%4];"
                     : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
                     : "r"(stage_base + 16u * static_cast<uint32_t>(p)));
        const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
        for (int e = 0; e < 8; ++e) {
          const uint16_t h = static_cast<uint16_t>(e & 1 ? (w[e >> 1] >> 16) : w[e >> 1]);
          asm volatile("st.shared.u16 [%0], %1;" ::"r"(dst[u][e]), "h"(h) : "memory");
        }
      }
    }
    __syncthreads();
    // raw stage s is free again: refill it with the tile `stages` ahead
    if (tid == 0) refill(s);

    // ---- phase 2: block Walsh-Hadamard transform and row abs-max ----------
    float2 v[16];  // v[k] holds positions 2k, 2k+1 of the segment
#pragma unroll
    for (int c = 0; c < 4; ++c) {
      uint4 raw4;
      asm volatile("ld.shared.v4.u32 {%0,%1,%2,%3}, [%4];"
                   : "=r"(raw4.x), "=r"(raw4.y), "=r"(raw4.z), "=r"(raw4.w)
                   : "r"(seg_addr[c])
                   : "memory");
      v[4 * c + 0] = to_f2<T>(raw4.x);
      v[4 * c + 1] = to_f2<T>(raw4.y);
      v[4 * c + 2] = to_f2<T>(raw4.z);
      v[4 * c + 3] = to_f2<T>(raw4.w);
    }
    const float2 neg1 = make_float2(-1.f, -1.f);
    if (lb >= 1) {  // stride 1: inside each pair
#pragma unroll
      for (int k = 0; k < 16; ++k) v[k] = make_float2(v[k].x + v[k].y, v[k].x - v[k].y);
    }
    // strides 2 .. min(b, 32) / 2: whole pairs k and k + h / 2
#pragma unroll
    for (int hp = 1; hp < 16; hp <<= 1) {
      if (2 * hp < (1 << lb)) {
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
    // strides 32 .. b / 2 across lanes: partner lane = lane ^ hl
#pragma unroll
    for (int hl = 1; hl < 8; hl <<= 1) {
      if (lb > 5 && hl < (1 << (lb > 5 ? lb - 5 : 0))) {
        const float sg = (lane & hl) ? -1.f : 1.f;
        const float2 sg2 = make_float2(sg, sg);
#pragma unroll
        for (int k = 0; k < 16; ++k) {
          float2 p;
          p.x = __shfl_xor_sync(0xffffffffu, v[k].x, hl);
          p.y = __shfl_xor_sync(0xffffffffu, v[k].y, hl);
          v[k] = __ffma2_rn(v[k], sg2, p);  // lower: x + p, upper: p - x
        }
      }
    }
    float m = 0.f;
#pragma unroll
    for (int k = 0; k < 16; ++k) m = fmaxf(m, fmaxf(fabsf(v[k].x), fabsf(v[k].y)));
    // Lanes of this warp on the same row; padding lanes (tid >= items) only
    // keep the shuffles convergent, their values are not data of any row and
    // must not reach a row maximum.
    const unsigned grp = __match_any_sync(0xffffffffu, active ? r_local : -1);
    const int leader = __ffs(grp) - 1;
    {
      const unsigned mx = __reduce_max_sync(grp, __float_as_uint(m));
      if (active && lane == leader) atomicMax(&sh.amax[par * R + r_local], mx);
    }
    __syncthreads();

    // ---- phase 3: scale, codes, pack, store --------------------------------
    if (active && r_local < rows) {
      const int row = row0 + r_local;
      // One lane per (row, warp) computes the scale and its reciprocal.
      float s_row = 0.f, rcp = 0.f;
      if (lane == leader) {
        float amax = __uint_as_float(sh.amax[par * R + r_local]);
        if (CLIP) amax = fminf(amax, __ldg(a.clip + row));
        s_row = __fdiv_rn(amax, 7.0f);
        rcp = s_row > 0.f ? __frcp_rn(s_row) : 0.f;
      }
      s_row = __shfl_sync(grp, s_row, leader);
      rcp = __shfl_sync(grp, rcp, leader);
      const float2 rc2 = make_float2(rcp, rcp);
      const float2 magic = make_float2(12582912.0f, 12582912.0f);  // 1.5 * 2^23
      if (a.e4m3) {
        // one byte per code: the E4M3 encoding of the integer code
        uint32_t w[8];
#pragma unroll
        for (int k = 0; k < 16; k += 2) {
          uint32_t h[2];
#pragma unroll
          for (int j = 0; j < 2; ++j) {
            float2 r = __fmul2_rn(v[k + j], rc2);
            if (CLIP) {
              r.x = fminf(fmaxf(r.x, -7.f), 7.f);
              r.y = fminf(fmaxf(r.y, -7.f), 7.f);
            }
            const float2 q = __fadd2_rn(__fadd2_rn(r, magic), make_float2(-12582912.0f, -12582912.0f));
            uint16_t e;
            asm("cvt.rn.satfinite.e4m3x2.f32 %0, %1, %2;" : "=h"(e) : "f"(q.y), "f"(q.x));
            h[j] = e;
          }
          w[k >> 1] = h[0] | (h[1] << 16);
        }
        uint4* qrow = reinterpret_cast<uint4*>(a.Q + static_cast<size_t>(row) * K + seg * 32);
        qrow[0] = make_uint4(w[0], w[1], w[2], w[3]);
        qrow[1] = make_uint4(w[4], w[5], w[6], w[7]);
      } else {
        // two codes per byte: the low nibble of (x / s + 1.5 * 2^23)'s bits
        // is the code's two's complement
        uint32_t by[16];
#pragma unroll
        for (int k = 0; k < 16; ++k) {
          float2 r = __fmul2_rn(v[k], rc2);
          if (CLIP) {
            r.x = fminf(fmaxf(r.x, -7.f), 7.f);
            r.y = fminf(fmaxf(r.y, -7.f), 7.f);
          }
          const float2 t = __fadd2_rn(r, magic);
          const uint32_t b0 = __float_as_uint(t.x), b1 = __float_as_uint(t.y);
          by[k] = (b0 & 0xFu) | ((b1 << 4) & 0xF0u);
        }
        uint32_t w[4];
#pragma unroll
        for (int q = 0; q < 4; ++q)
          w[q] = prmt_b32(prmt_b32(by[4 * q], by[4 * q + 1], 0x0040u),
                          prmt_b32(by[4 * q + 2], by[4 * q + 3], 0x0040u), 0x5410u);
        uint8_t* qrow = a.Q + static_cast<size_t>(row) * (K >> 1);
        *reinterpret_cast<uint4*>(qrow + seg * 16) = make_uint4(w[0], w[1], w[2], w[3]);
      }
      if (seg == 0) a.S[row] = s_row;
      if (a.rot != nullptr) {
        float4* dst = reinterpret_cast<float4*>(a.rot + static_cast<size_t>(row) * K + seg * 32);
#pragma unroll
        for (int q = 0; q < 8; ++q)
          dst[q] = make_float4(v[2 * q].x, v[2 * q].y, v[2 * q + 1].x, v[2 * q + 1].y);
      }
    }
    if (tid < R) sh.amax[(par ^ 1) * R + tid] = 0u;
    publish(row0, rows);
  }

  // After an abort, copies already issued must land before the memory is
  // reused; then the barriers are invalidated so the buffer can be repurposed.
  if (tid == 0 && aborted) {
    for (int s = 0; s < stages; ++s)
      for (int ph = 0; ph < 2; ++ph)
        mbar_wait_bounded(&sh.full[s], ph, nullptr, nullptr, 10000000ull);
  }
  __syncthreads();
  if (tid == 0)
    for (int s = 0; s < stages; ++s) mbar_inval(&sh.full[s]);
}

}  // namespace rq
}  // namespace clq
