// Rotate-quantize tile loop, shared by the standalone kernel and the fused
// linear kernel.  It applies the OBS transform of arxiv 2509.24416 Sec. 3.3
// to rows of X (column gather by the swap vector `perm`, then the block
// Sylvester Hadamard H_b) and quantizes each row to symmetric INT4 with a
// dynamic fp32 scale (Sec. 3.1, Eq. 1 with l = -r), or to symmetric INT8
// (qmax 127) for the split-plane layout of the W4A8 / W8A8 settings, or
// (ASYM) asymmetrically with the row's min and max as bounds (Eq. 1 with
// dynamic l and r), stored as centered codes q - 2^(n-1).
//
// The standalone activation path with symmetric 4-bit codes in the E4M3 or
// E2M3 layout and b >= 32 runs the specialized loops of rq_pair.cuh and
// rq_wide.cuh; this general loop serves every other setting (packed codes,
// b < 32, 8-bit and asymmetric codes, clipped weights) and the fused kernel.
//
// Every thread of the CTA takes part.  The CTA walks tiles of R rows.  Raw
// rows stream into a ring of STAGES shared-memory buffers (STRIDE bytes
// apart, both compile-time, so that a stage's address is an immediate
// offset) with bulk asynchronous copies (cp.async.bulk + mbarrier), so
// several tiles are in flight per SM while the threads work on an earlier
// one.  Thread (row, segment) owns permuted positions 32 * segment .. + 31 of
// its row.  Per tile:
//  1. gather: each of the 32 elements is read straight from the raw stage at
//     column perm[position] (one 16-bit shared load; the 32 byte offsets are
//     computed once per CTA), and the first butterfly stage (stride 1) is
//     done on the way in with mixed-precision add / sub (one 16-bit operand,
//     one fp32 operand, fp32 result).  For the symmetric E4M3 output each
//     lane group reads its segment in the order position ^ m (m a multiple
//     of 8 that differs between neighbouring lane groups), which spreads the
//     lanes' 16-bit loads over the shared-memory banks (a swap vector is
//     mostly ascending, so in natural order the lanes of a warp hit the same
//     banks); see xor_order below for why the result only changes sign;
//  2. the remaining butterfly stages up to stride 16 in registers (paired
//     fp32x2 arithmetic), strides 32 .. b / 2 across lanes with shuffles,
//     then the row's |x| maximum: warp reduction and a shared atomicMax;
//  3. one CTA barrier; then s = absmax / qmax, codes rint(x / s) (x times an
//     approximate reciprocal of s, rounded with the 1.5 * 2^23 constant,
//     ties to even), stored as packed nibbles, one E4M3 byte per code, or
//     (8 bits) two E4M3 planes 16 h and l with q = 16 h + l, l in [-8, 7].
// The row maxima are triple-buffered over tiles, so the barrier of tile i
// also separates the readers of tile i - 1 from the reset for tile i + 2.
#pragma once

#include "clq_device.cuh"
#include "clq_kernels.h"

namespace clq {
namespace rq {

// Stage geometry of the standalone kernel: two stages of 32 KB (a tile of R
// rows of K 16-bit elements, 2 R K bytes, fits one stage for every K up to
// 16384).  Measured against 16 KB x 4, 16 KB x 3 and 24 KB x 3: 2-7 % faster
// (a shorter unrolled stage loop, more rows per tile available).
constexpr int kStride = 32 * 1024;
constexpr int kStages = 2;
constexpr int kMaxRegs = 128;            // register cap of the tile-loop kernels

// Shared memory of the tile loop: STAGES raw tiles, 3R row maxima and 3R row
// minima (asymmetric mode), 2 x STAGES barriers, STAGES tile indices, abort
// flag.
__host__ __device__ inline size_t smem_bytes(int R, int stride, int stages) {
  return static_cast<size_t>(stages) * stride + 24u * R + 8u + 20u * stages + 16u;
}

// Order-preserving map of a float to an unsigned key (and back), so that
// signed maxima can be taken with integer max reductions; key 0 is below
// every float.
__device__ __forceinline__ uint32_t order_key(float f) {
  const uint32_t u = __float_as_uint(f);
  return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}
__device__ __forceinline__ float order_key_inv(uint32_t k) {
  return __uint_as_float((k & 0x80000000u) ? (k & 0x7FFFFFFFu) : ~k);
}

// Publish policy of the tile loop.  operator(): called by every thread of
// the team once its stores of a tile are issued.  release(): called by the
// loader thread only (loader mode), after every compute thread has fenced its
// stores of the tile for the async proxy and signalled it.
struct NoPublish {
  __device__ void operator()(int, int) const {}
  __device__ void release(int, int) const {}
};

// The threads that run the tile loop: the whole CTA (count 0, barrier id 0:
// __syncthreads) or `count` threads from thread `first` on (whole warps)
// synchronized by named barrier `bar`, while other warps of the CTA do other
// work.  In loader mode the last warp of the team is the loader, the others
// compute and synchronize by barrier `bar`; barrier `bar + 1` spans the team.
struct Team {
  int first = 0;
  int count = 0;
  uint32_t bar = 0;
  __device__ int size() const { return count > 0 ? count : static_cast<int>(blockDim.x); }
  __device__ int rank() const { return static_cast<int>(threadIdx.x) - first; }
  __device__ void sync() const {
    if (bar == 0)
      __syncthreads();
    else
      asm volatile("bar.sync %0, %1;" ::"r"(bar), "r"(count) : "memory");
  }
};

// One 16-bit value -> fp32, exactly.
template <typename T>
__device__ __forceinline__ float to_f32(uint16_t h);
template <>
__device__ __forceinline__ float to_f32<__half>(uint16_t h) {
  return __half2float(__ushort_as_half(h));
}
template <>
__device__ __forceinline__ float to_f32<__nv_bfloat16>(uint16_t h) {
  return __uint_as_float(static_cast<uint32_t>(h) << 16);
}

// (a + b, a - b) in fp32 from a 16-bit a and an fp32 b (one rounding each).
template <typename T>
__device__ __forceinline__ float2 add_sub_mixed(uint16_t a, float b);
template <>
__device__ __forceinline__ float2 add_sub_mixed<__half>(uint16_t a, float b) {
  float s, d;
  asm("add.rn.f32.f16 %0, %1, %2;" : "=f"(s) : "h"(a), "f"(b));
  asm("sub.rn.f32.f16 %0, %1, %2;" : "=f"(d) : "h"(a), "f"(b));
  return make_float2(s, d);
}
template <>
__device__ __forceinline__ float2 add_sub_mixed<__nv_bfloat16>(uint16_t a, float b) {
  float s, d;
  asm("add.rn.f32.bf16 %0, %1, %2;" : "=f"(s) : "h"(a), "f"(b));
  asm("sub.rn.f32.bf16 %0, %1, %2;" : "=f"(d) : "h"(a), "f"(b));
  return make_float2(s, d);
}

// Shared-memory 16-bit load.  Volatile: the raw stages are rewritten by the
// bulk copies between tiles, which the compiler cannot see.
__device__ __forceinline__ uint16_t lds_u16(uint32_t addr) {
  uint16_t v;
  asm volatile("ld.shared.b16 %0, [%1];" : "=h"(v) : "r"(addr) : "memory");
  return v;
}

__device__ __forceinline__ uint32_t prmt_b32(uint32_t a, uint32_t b, uint32_t c) {
  uint32_t d;
  asm("prmt.b32 %0, %1, %2, %3;" : "=r"(d) : "r"(a), "r"(b), "r"(c));
  return d;
}

// Approximate reciprocal (hardware, within one unit in the last place) of a
// normal positive float.
__device__ __forceinline__ float rcp_approx(float x) {
  float r;
  asm("rcp.approx.ftz.f32 %0, %1;" : "=f"(r) : "f"(x));
  return r;
}

__device__ __forceinline__ void mbar_inval(uint64_t* bar) {
  asm volatile("mbarrier.inval.shared::cta.b64 [%0];" ::"r"(smem_addr(bar)) : "memory");
}

// Issue the bulk copies of tile `tile` into the raw stage at `dst`.
__device__ __forceinline__ void issue_tile(const RotateQuantArgs& a, uint8_t* dst, uint64_t* bar,
                                           int R, int tile) {
  const int row0 = tile * R;
  const int rows = min(R, a.M - row0);
  const uint32_t row_bytes = static_cast<uint32_t>(a.K) * 2u;
  const char* src = static_cast<const char*>(a.X) + static_cast<size_t>(row0) * a.ld * 2u;
  mbar_arrive_expect_tx(bar, row_bytes * rows);
  if (a.ld == a.K) {
    bulk_load(dst, src, row_bytes * rows, bar);
  } else {
    for (int r = 0; r < rows; ++r)
      bulk_load(dst + static_cast<size_t>(r) * row_bytes,
                src + static_cast<size_t>(r) * a.ld * 2u, row_bytes, bar);
  }
}

// Runs the tile loop with every thread of the CTA, or with the threads of
// `team` (R * K / 32 <= its compute threads, 2 R K <= STRIDE).  Tiles come in
// a static round-robin order (tile_counter == null) or are claimed one at a
// time from a global counter (so that CTAs which never become resident own
// no rows).  After each tile, every thread
// calls publish(row0, rows) once its own stores of that tile are issued.
// LOGB = log2(b) when known at compile time, or -1 to read a.logb.  SPLIT:
// 8-bit codes in the split-plane layout (a.e4m3 == 2), else 4-bit codes.
// ASYM: asymmetric codes with per-row a.S = delta and a.lo = min.
//
// LOADER (needs a Team with count > 32 and bar != 0): one warp of the team
// takes every step whose latency is global off the compute warps: it claims
// tiles one ahead of their refill, refills the stages, and publishes a tile
// (publish.release) once the compute warps have signalled its stores on the
// stage's `done` barrier.  The compute warps then only wait for their data.
template <typename T, int LOGB, bool CLIP, int STRIDE, int STAGES, bool SPLIT = false,
          bool ASYM = false, typename Publish = NoPublish, bool LOADER = false>
__device__ __forceinline__ void run(const RotateQuantArgs& a, uint8_t* smem,
                                    uint32_t* tile_counter, Publish publish,
                                    Team team = Team()) {
  const int K = a.K;
  const int segs = K >> 5;
  const int R = a.rows_per_tile;
  const int lb = LOGB >= 0 ? LOGB : a.logb;  // log2(b): compile time or runtime
  const int nthr = LOADER ? team.count - 32 : team.size();  // compute threads
  const int tid = team.rank();
  // compute threads only (loader mode), every team thread
  auto csync = [&]() {
    if (LOADER)
      asm volatile("bar.sync %0, %1;" ::"r"(team.bar), "r"(nthr) : "memory");
    else
      team.sync();
  };
  auto tsync = [&]() {
    if (LOADER)
      asm volatile("bar.sync %0, %1;" ::"r"(team.bar + 1), "r"(team.count) : "memory");
    else
      team.sync();
  };
  const int lane = tid & 31;
  const uint32_t row_bytes = static_cast<uint32_t>(K) * 2u;

  uint8_t* raw = smem;
  uint32_t* amax = reinterpret_cast<uint32_t*>(smem + STAGES * STRIDE);  // [3][R]
  uint32_t* amin = amax + 3 * R;  // [3][R] keys of -min (asymmetric mode)
  uint64_t* full = reinterpret_cast<uint64_t*>(
      (reinterpret_cast<uintptr_t>(amin + 3 * R) + 7) & ~static_cast<uintptr_t>(7));
  uint64_t* done_bar = full + STAGES;  // loader mode: the stage's tile is stored
  int32_t* tile_of = reinterpret_cast<int32_t*>(done_bar + STAGES);  // tile in each stage
  int32_t* abort = tile_of + STAGES;

  const int ntiles = (a.M + R - 1) / R;
  int claims = 0;  // refilling thread: tiles claimed so far
  int ahead = 0;   // loader: the tile claimed for the next refill
  // tid 0 (the loader thread in loader mode): claim the next tile into stage
  // s and start its copies (or mark the stage empty and complete its phase
  // without data).  Past the first STAGES claims, which every CTA makes one
  // at a time so that the first tiles of all CTAs are the lowest rows, the
  // loader claims one tile ahead: the atomic's round trip then overlaps the
  // wait for the next stage.
  auto refill = [&](int s) {
    int t;
    if (tile_counter != nullptr) {
      if (LOADER && claims >= STAGES) {
        t = ahead;
        ahead = static_cast<int>(atomicAdd(tile_counter, 1u));
      } else {
        t = static_cast<int>(atomicAdd(tile_counter, 1u));
      }
    } else {
      t = static_cast<int>(blockIdx.x) + claims * static_cast<int>(gridDim.x);
    }
    ++claims;
    if (t < ntiles) {
      tile_of[s] = t;
      issue_tile(a, raw + s * STRIDE, &full[s], R, t);
    } else {
      tile_of[s] = -1;
      mbar_arrive(&full[s]);
    }
  };

  if (tid == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&done_bar[s], nthr / 32);
    }
    *abort = 0;
    fence_mbarrier_init();
  }
  for (int i = tid; i < 6 * R; i += team.size()) amax[i] = 0u;
  // Round-robin tiles: this CTA's first tiles into L2 while the previous
  // kernel drains; the copies after the wait still read every value from L2 /
  // memory, where the previous kernel's writes land.
  if (tid == 0 && tile_counter == nullptr && a.ld == a.K)
    for (int s = 0; s < STAGES; ++s) {
      const int t = static_cast<int>(blockIdx.x) + s * static_cast<int>(gridDim.x);
      if (t < ntiles) {
        const int row0 = t * R;
        const uint32_t row_bytes = static_cast<uint32_t>(a.K) * 2u;
        bulk_prefetch_l2(static_cast<const char*>(a.X) + static_cast<size_t>(row0) * row_bytes,
                         row_bytes * static_cast<uint32_t>(min(R, a.M - row0)));
      }
    }
  tsync();
  // Past pdl_wait, the previous kernel on the stream has completed (it may
  // still be finishing when this grid starts): X, the tile counter and every
  // output are touched only after it, the swap vector (a layer constant that
  // no kernel of this library writes) before it.
  if (LOADER && tid >= nthr) {
    // ---- loader warp ---------------------------------------------------------
    pdl_wait();
    pdl_launch_dependents();
    if ((tid & 31) == 0) {
      for (int s = 0; s < STAGES; ++s) refill(s);
      if (tile_counter != nullptr) ahead = static_cast<int>(atomicAdd(tile_counter, 1u));
      for (int j = 0;; ++j) {
        const int s = j % STAGES;
        const int tile = *reinterpret_cast<volatile int32_t*>(&tile_of[s]);
        if (tile < 0) break;
        if (!mbar_wait_bounded(&done_bar[s], (j / STAGES) & 1, abort, a.status, kWaitLimitNs))
          break;
        publish.release(tile * R, min(R, a.M - tile * R));
        refill(s);
      }
      // After an abort, copies already issued must land before the memory
      // is reused.
      if (*reinterpret_cast<volatile int32_t*>(abort) != 0)
        for (int s = 0; s < STAGES; ++s)
          for (int ph = 0; ph < 2; ++ph)
            mbar_wait_bounded(&full[s], ph, nullptr, nullptr, 10000000ull);
    }
    __syncwarp();
  } else {
    const int items = R * segs;
    const bool active = tid < items;
    const int r_local = active ? tid / segs : 0;
    const int seg = active ? tid - r_local * segs : 0;
    // Shared addresses (stage 0) of this thread's 32 elements: column
    // perm[32 seg + k] of row r_local.  An index outside [0, K) is reported and
    // replaced by column 0, so a bad swap vector gives wrong values, never a
    // stray access.
    uint32_t src[32];
    // xor_order: register k holds segment position k ^ m.  The butterflies
    // then compute H_b P_m x, and since H[i][j ^ m] = (-1)^popc(i & m) H[i][j]
    // for Sylvester H, that is D_m H_b x with D_m = diag((-1)^popc(i & m)):
    // the transform up to a sign per output.  Lanes combined by the
    // cross-lane stages share m, so the signs factor out of those stages too.
    // The row maximum ignores signs; the codes get them back when stored (for
    // m a multiple of 4 the sign is the same for the 4 codes of one 32-bit
    // word: bit q of flip_words).  Only the symmetric E4M3 path uses it, with
    // m a multiple of 8 (b >= 16): measured faster than multiples of 4, 16 or
    // masks with low bits, which break up the 4-byte bank words that adjacent
    // columns share.
    const bool xor_order = (a.e4m3 == 1 || a.e4m3 == 3) && !CLIP && !SPLIT && !ASYM && lb >= 4 &&
                           (reinterpret_cast<uintptr_t>(a.perm) & 15u) == 0;
    const int xm = xor_order ? ((8 * (lane >> (lb > 5 ? lb - 5 : 0))) &
                                ((1 << (lb < 5 ? lb : 5)) - 8))
                             : 0;
    uint32_t flip_words = 0;
#pragma unroll
    for (int q = 0; q < 8; ++q)
      if (__popc(q & (xm >> 2)) & 1) flip_words |= 1u << q;
    {
      const uint32_t base = smem_addr(raw) + static_cast<uint32_t>(r_local) * row_bytes;
      int pc[32];
      const int32_t* pp = a.perm + seg * 32;
      if ((reinterpret_cast<uintptr_t>(a.perm) & 15u) == 0) {  // 16-byte loads
#pragma unroll
        for (int q = 0; q < 8; ++q) {
          const int4 t = active ? __ldg(reinterpret_cast<const int4*>(pp) + (q ^ (xm >> 2)))
                                : make_int4(0, 0, 0, 0);
          pc[4 * q] = t.x;
          pc[4 * q + 1] = t.y;
          pc[4 * q + 2] = t.z;
          pc[4 * q + 3] = t.w;
        }
      } else {
#pragma unroll
        for (int k = 0; k < 32; ++k) pc[k] = active ? __ldg(pp + k) : 0;
      }
      bool bad = false;
#pragma unroll
      for (int k = 0; k < 32; ++k) {
        const bool out = static_cast<unsigned>(pc[k]) >= static_cast<unsigned>(K);
        bad |= out;
        src[k] = base + 2u * static_cast<uint32_t>(out ? 0 : pc[k]);
      }
      if (bad) record_status(a.status, CLQ_ERR_DEVICE_INDEX);
    }
    // Lanes of this warp on the same row (fixed for the whole launch).  Padding
    // lanes (tid >= items) only keep the shuffles convergent; their values are
    // not data of any row and must not reach a row maximum.
    const unsigned grp = __match_any_sync(0xffffffffu, active ? r_local : -1);
    const int leader = __ffs(grp) - 1;
    pdl_wait();
    pdl_launch_dependents();
    if (!LOADER && tid == 0)
      for (int s = 0; s < STAGES; ++s) refill(s);

    bool aborted = false, done = false;
    for (int i0 = 0; !done; i0 += STAGES) {
#pragma unroll
      for (int s = 0; s < STAGES; ++s) {
        if (done) break;
        const int i = i0 + s;
        if (!mbar_wait_bounded(&full[s], (i0 / STAGES) & 1, abort, a.status, kWaitLimitNs)) {
          aborted = done = true;
          break;
        }
        const int tile = *reinterpret_cast<volatile int32_t*>(&tile_of[s]);
        if (tile < 0) {
          done = true;
          break;
        }
        const int row0 = tile * R;
        const int rows = min(R, a.M - row0);
        const int par = i % 3;

        // ---- 1. gather + first butterfly stage --------------------------------
        float2 v[16];  // v[k] holds positions 2k, 2k+1 of the segment
#pragma unroll
        for (int k = 0; k < 16; ++k) {
          const uint16_t x0 = lds_u16(src[2 * k] + s * STRIDE);
          const uint16_t x1 = lds_u16(src[2 * k + 1] + s * STRIDE);
          if (lb >= 1)
            v[k] = add_sub_mixed<T>(x0, to_f32<T>(x1));
          else
            v[k] = make_float2(to_f32<T>(x0), to_f32<T>(x1));
        }

        // ---- 2. remaining butterfly stages and row abs-max --------------------
        const float2 neg1 = make_float2(-1.f, -1.f);
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
        if constexpr (ASYM) {
          // max and min of the segment as trees, reduced as order keys
          float mk[16];
#pragma unroll
          for (int k = 0; k < 16; ++k) mk[k] = fmaxf(v[k].x, v[k].y);
#pragma unroll
          for (int w = 8; w >= 1; w >>= 1)
#pragma unroll
            for (int k = 0; k < w; ++k) mk[k] = fmaxf(mk[k], mk[k + w]);
          const unsigned kx = __reduce_max_sync(grp, order_key(mk[0]));
#pragma unroll
          for (int k = 0; k < 16; ++k) mk[k] = fminf(v[k].x, v[k].y);
#pragma unroll
          for (int w = 8; w >= 1; w >>= 1)
#pragma unroll
            for (int k = 0; k < w; ++k) mk[k] = fminf(mk[k], mk[k + w]);
          const unsigned kn = __reduce_max_sync(grp, order_key(-mk[0]));
          if (active && lane == leader && r_local < rows) {
            atomicMax(&amax[par * R + r_local], kx);
            atomicMax(&amin[par * R + r_local], kn);
          }
        } else {
          // |x| maximum of the segment as a tree (short dependency chain)
          float mk[16];
#pragma unroll
          for (int k = 0; k < 16; ++k) mk[k] = fmaxf(fabsf(v[k].x), fabsf(v[k].y));
#pragma unroll
          for (int w = 8; w >= 1; w >>= 1)
#pragma unroll
            for (int k = 0; k < w; ++k) mk[k] = fmaxf(mk[k], mk[k + w]);
          const unsigned mx = __reduce_max_sync(grp, __float_as_uint(mk[0]));
          if (active && lane == leader && r_local < rows) atomicMax(&amax[par * R + r_local], mx);
        }
        csync();  // row maxima complete; raw stage s fully read
        if (!LOADER && tid == 0) refill(s);

        // ---- 3. scale, codes, pack, store --------------------------------------
        if (active && r_local < rows) {
          const int row = row0 + r_local;
          constexpr float qmax = SPLIT ? 127.0f : 7.0f;
          float am, row_lo = 0.f;
          if constexpr (ASYM) {
            // span = max - min; delta = span / (2^n - 1)
            row_lo = -order_key_inv(amin[par * R + r_local]);
            am = __fsub_rn(order_key_inv(amax[par * R + r_local]), row_lo);
          } else {
            am = __uint_as_float(amax[par * R + r_local]);
            if (CLIP) am = fminf(am, __ldg(a.clip + row));
          }
          // s = am / qmax (symmetric) or am / (2 qmax + 1) (asymmetric), by
          // division by a constant known in advance (Brisebarre, Muller and
          // Raina, IEEE Trans. Computers 53(8), 2004): q1 = RN(am * RN(1/d)),
          // the exact residual am - d q1 by one fma, and one more fma that
          // adds residual * RN(1/d) back to q1; within one ulp of the IEEE
          // quotient for every am (tested against it).
          constexpr float div = ASYM ? 2.0f * qmax + 1.0f : qmax;
          constexpr float rdiv = 1.0f / div;
          const float q1 = am * rdiv;
          const float s_row = fmaf(fmaf(-div, q1, am), rdiv, q1);
          if (seg == 0) {
            a.S[row] = s_row;
            if (ASYM) a.lo[row] = row_lo;
          }
          if (a.rot != nullptr) {
            float4* dst =
                reinterpret_cast<float4*>(a.rot + static_cast<size_t>(row) * K + seg * 32);
#pragma unroll
            for (int q = 0; q < 8; ++q) {
              const float sg = ((flip_words >> q) & 1u) ? -1.f : 1.f;
              dst[q] = make_float4(sg * v[2 * q].x, sg * v[2 * q].y, sg * v[2 * q + 1].x,
                                   sg * v[2 * q + 1].y);
            }
          }
          // v <- rint(v / s) + 1.5 * 2^23 (the code sits in the low mantissa
          // bits), with v / s as v * (1 / s).  A zero row (s = 0) gets all-zero
          // codes; a subnormal s (a row maximum below about 1e-37) takes exact
          // divisions instead of the reciprocal.
          const float2 magic = make_float2(12582912.0f, 12582912.0f);  // 1.5 * 2^23
          if constexpr (ASYM) {
            // q = rint((x - min) / span * (2^n - 1)), stored as q - 2^(n-1): the
            // magic constant is lowered by 2^(n-1) (it stays even, so ties
            // still go to even q).  A constant row (span 0) gets q = 0.
            constexpr float half = SPLIT ? 128.0f : 8.0f;
            const float2 mg = make_float2(12582912.0f - half, 12582912.0f - half);
            const float2 nlo = make_float2(-row_lo, -row_lo);
            // exact divisions also where rcp(span) would be subnormal (span
            // >= 2^126, bf16 inputs near their top), which rcp.approx.ftz
            // flushes to zero
            if (am > 0.f && (am < 1.17549435e-38f || am >= 8.50705917e37f)) {
#pragma unroll
              for (int k = 0; k < 16; ++k) {
                const float2 d = __fadd2_rn(v[k], nlo);
                v[k] = __fadd2_rn(make_float2(__fmul_rn(__fdiv_rn(d.x, am), div),
                                              __fmul_rn(__fdiv_rn(d.y, am), div)),
                                  mg);
              }
            } else {
              const float inv = am > 0.f ? div * rcp_approx(am) : 0.f;
              const float2 inv2 = make_float2(inv, inv);
#pragma unroll
              for (int k = 0; k < 16; ++k) v[k] = __ffma2_rn(__fadd2_rn(v[k], nlo), inv2, mg);
            }
          } else if (s_row > 0.f && s_row < 1.17549435e-38f) {
#pragma unroll
            for (int k = 0; k < 16; ++k)
              v[k] = __fadd2_rn(make_float2(__fdiv_rn(v[k].x, s_row), __fdiv_rn(v[k].y, s_row)),
                                magic);
          } else {
            const float rcp = s_row > 0.f ? rcp_approx(s_row) : 0.f;
            const float2 rc2 = make_float2(rcp, rcp);
#pragma unroll
            for (int k = 0; k < 16; ++k) v[k] = __ffma2_rn(v[k], rc2, magic);
          }
          if (CLIP) {  // clipped weight rows: |v / s| may exceed qmax
            const float lo = 12582912.0f - qmax, hi = 12582912.0f + qmax;
#pragma unroll
            for (int k = 0; k < 16; ++k) {
              v[k].x = fminf(fmaxf(v[k].x, lo), hi);
              v[k].y = fminf(fmaxf(v[k].y, lo), hi);
            }
          }
          if constexpr (SPLIT) {
            // q = 16 h + l with h = floor((q + 8) / 16): plane 0 gets the E4M3
            // encoding of 16 h (a multiple of 16 in [-128, 128]), plane 1 that
            // of l in [-8, 7]; every step is exact in fp32.
            uint32_t wh[8], wl[8];
#pragma unroll
            for (int k = 0; k < 16; k += 2) {
              uint32_t hh[2], ll[2];
#pragma unroll
              for (int j = 0; j < 2; ++j) {
                const float2 q = __fadd2_rn(v[k + j], make_float2(-12582912.0f, -12582912.0f));
                const float2 t = __fmul2_rn(__fadd2_rn(q, make_float2(8.f, 8.f)),
                                            make_float2(0.0625f, 0.0625f));
                const float2 h16 = make_float2(16.f * floorf(t.x), 16.f * floorf(t.y));
                const float2 l = __fadd2_rn(q, make_float2(-h16.x, -h16.y));
                uint16_t eh, el;
                asm("cvt.rn.satfinite.e4m3x2.f32 %0, %1, %2;" : "=h"(eh) : "f"(h16.y), "f"(h16.x));
                asm("cvt.rn.satfinite.e4m3x2.f32 %0, %1, %2;" : "=h"(el) : "f"(l.y), "f"(l.x));
                hh[j] = eh;
                ll[j] = el;
              }
              wh[k >> 1] = hh[0] | (hh[1] << 16);
              wl[k >> 1] = ll[0] | (ll[1] << 16);
            }
            uint4* qh = reinterpret_cast<uint4*>(a.Q + static_cast<size_t>(row) * 2 * K + seg * 32);
            uint4* ql = reinterpret_cast<uint4*>(a.Q + (static_cast<size_t>(row) * 2 + 1) * K +
                                                 seg * 32);
            qh[0] = make_uint4(wh[0], wh[1], wh[2], wh[3]);
            qh[1] = make_uint4(wh[4], wh[5], wh[6], wh[7]);
            ql[0] = make_uint4(wl[0], wl[1], wl[2], wl[3]);
            ql[1] = make_uint4(wl[4], wl[5], wl[6], wl[7]);
          } else if (a.e4m3 == 3) {
            // E2M3 codes, 16 to 12 bytes: each group of 16 consecutive codes
            // is one little-endian 96-bit field, code i in bits 6i .. 6i + 5.
            // cvt gives each code's 6-bit encoding in a byte (sign bit 5); four
            // of those bytes c = b0 | b1 << 8 | b2 << 16 | b3 << 24 close up to
            // 24 bits by two subtractions: c - 3 (b1 << 6 | b3 << 22) moves b1
            // and b3 down two bits, t - 15 (hi << 12) moves the upper 12-bit
            // pair down four.
            uint32_t g[8];
#pragma unroll
            for (int k = 0; k < 16; k += 2) {
              uint32_t h[2];
#pragma unroll
              for (int j = 0; j < 2; ++j) {
                const float2 q = __fadd2_rn(v[k + j], make_float2(-12582912.0f, -12582912.0f));
                uint16_t e;
                asm("cvt.rn.satfinite.e2m3x2.f32 %0, %1, %2;" : "=h"(e) : "f"(q.y), "f"(q.x));
                h[j] = e;
              }
              uint32_t c = h[0] | (h[1] << 16);
              c ^= (0u - ((flip_words >> (k >> 1)) & 1u)) & 0x20202020u;  // xor_order signs
              const uint32_t t = c - 3u * ((c >> 2) & 0x0FC00FC0u);
              g[k >> 1] = t - 15u * ((t >> 4) & 0x00FFF000u);
            }
            uint2* qrow = reinterpret_cast<uint2*>(a.Q + static_cast<size_t>(row) * (3 * K / 4) +
                                                   seg * 24);
            qrow[0] = make_uint2(g[0] | (g[1] << 24), (g[1] >> 8) | (g[2] << 16));
            qrow[1] = make_uint2((g[2] >> 16) | (g[3] << 8), g[4] | (g[5] << 24));
            qrow[2] = make_uint2((g[5] >> 8) | (g[6] << 16), (g[6] >> 16) | (g[7] << 8));
          } else if (a.e4m3) {
            // one byte per code: the E4M3 encoding of the integer code
            uint32_t w[8];
#pragma unroll
            for (int k = 0; k < 16; k += 2) {
              uint32_t h[2];
#pragma unroll
              for (int j = 0; j < 2; ++j) {
                const float2 q = __fadd2_rn(v[k + j], make_float2(-12582912.0f, -12582912.0f));
                uint16_t e;
                asm("cvt.rn.satfinite.e4m3x2.f32 %0, %1, %2;" : "=h"(e) : "f"(q.y), "f"(q.x));
                h[j] = e;
              }
              w[k >> 1] = h[0] | (h[1] << 16);
            }
            // xor_order signs back: flip the sign bit of each E4M3 byte of the
            // flagged words (a zero code may come out as E4M3 -0, 0x80)
#pragma unroll
            for (int q = 0; q < 8; ++q) w[q] ^= (0u - ((flip_words >> q) & 1u)) & 0x80808080u;
            uint4* qrow = reinterpret_cast<uint4*>(a.Q + static_cast<size_t>(row) * K + seg * 32);
            qrow[0] = make_uint4(w[0], w[1], w[2], w[3]);
            qrow[1] = make_uint4(w[4], w[5], w[6], w[7]);
          } else {
            // two codes per byte: the low nibble of the bits is the code's
            // two's complement
            uint32_t by[16];
#pragma unroll
            for (int k = 0; k < 16; ++k) {
              const uint32_t b0 = __float_as_uint(v[k].x), b1 = __float_as_uint(v[k].y);
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
        }
        if (tid < R) {
          amax[((i + 2) % 3) * R + tid] = 0u;
          if (ASYM) amin[((i + 2) % 3) * R + tid] = 0u;
        }
        if constexpr (LOADER) {
          // the stores of this tile become visible to the async proxy (the
          // GEMM's tensor loads) through the loader's release
          asm volatile("fence.proxy.async.global;" ::: "memory");
          __syncwarp();
          if (lane == 0) mbar_arrive(&done_bar[s]);
        } else {
          publish(row0, rows);
        }
      }
    }

    // After an abort, copies already issued must land before the memory is
    // reused; then the barriers are invalidated so the buffer can be repurposed.
    if (!LOADER && tid == 0 && aborted) {
      for (int s = 0; s < STAGES; ++s)
        for (int ph = 0; ph < 2; ++ph)
          mbar_wait_bounded(&full[s], ph, nullptr, nullptr, 10000000ull);
    }
  }  // compute threads
  tsync();
  if (tid == 0)
    for (int s = 0; s < STAGES; ++s) {
      mbar_inval(&full[s]);
      mbar_inval(&done_bar[s]);
    }
}

}  // namespace rq
}  // namespace clq
