// Rotate-quantize kernel: one HBM pass that applies the OBS transform of
// arxiv 2509.24416 Sec. 3.3 to rows of X (column gather by the swap vector
// `perm`, then the block Sylvester Hadamard H_b) and quantizes each row to
// symmetric INT4 with a dynamic fp32 scale (Sec. 3.1, Eq. 1 with l = -r).
// The same kernel prepares weights offline (per-output-channel scales with
// an optional clip bound).
//
// Work split.  A CTA owns R rows at a time ("tile") and one item per thread:
// item = (row, segment of 32 consecutive permuted positions).
//  phase 1: coalesced 16-byte loads of the R rows; each element is written
//           to its permuted position in a shared-memory row buffer
//           (scatter through the inverse of perm, built once per CTA);
//  phase 2: each thread reads its 32 positions (4 x 16 B, bank-conflict-free
//           thanks to a chunk swizzle), runs the first log2(min(b, 32))
//           butterfly stages in registers and the remaining log2(b / 32)
//           stages across lanes with shuffles, and reduces |x| per row;
//  phase 3: scale, codes, nibble packing, one 16-byte store per thread.
#include "clq_device.cuh"
#include "clq_kernels.h"

namespace clq {

namespace {

// Byte offset of permuted position j inside a row buffer.  16-byte chunk q
// is stored at q ^ ((q >> 3) & 3): a thread reading chunks 4s..4s+3 and its
// neighbours reading theirs hit distinct banks within every 8-lane phase.
__device__ __forceinline__ uint32_t rowbuf_offset(uint32_t j) {
  const uint32_t q = j >> 3;
  const uint32_t phys = q ^ ((q >> 3) & 3u);
  return (phys << 4) | ((j & 7u) << 1);
}

__device__ __forceinline__ uint4 ld_stream_v4(const void* p) {
  uint4 v;
  asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
               : "l"(p));
  return v;
}

template <typename T>
__device__ __forceinline__ void unpack8(const uint4& raw, float* out) {
  const uint32_t w[4] = {raw.x, raw.y, raw.z, raw.w};
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    out[2 * i] = Num<T>::to_f(static_cast<uint16_t>(w[i] & 0xFFFFu));
    out[2 * i + 1] = Num<T>::to_f(static_cast<uint16_t>(w[i] >> 16));
  }
}

template <typename T, int LOGB>
__global__ void __launch_bounds__(512) rotate_quant_kernel(RotateQuantArgs a) {
  extern __shared__ __align__(16) uint8_t smem[];
  const int K = a.K;
  const int segs = K >> 5;
  const int R = a.rows_per_tile;
  const int nthr = blockDim.x;
  const int tid = threadIdx.x;
  const int lane = tid & 31;

  uint16_t* dst_off = reinterpret_cast<uint16_t*>(smem);               // [K]
  uint8_t* rowbuf = smem + ((2 * K + 15) & ~15);                       // [R][2K]
  uint32_t* amax_s = reinterpret_cast<uint32_t*>(rowbuf + 2 * R * K);  // [2][R]

  // Inverse of perm as destination offsets.  Entries default to 0 so that a
  // perm that is not a permutation produces wrong values, never a stray
  // shared-memory write; out-of-range indices are reported and skipped.
  for (int c = tid; c < K; c += nthr) dst_off[c] = 0;
  for (int i = tid; i < 2 * R; i += nthr) amax_s[i] = 0u;
  __syncthreads();
  for (int j = tid; j < K; j += nthr) {
    const int c = __ldg(a.perm + j);
    if (static_cast<unsigned>(c) < static_cast<unsigned>(K))
      dst_off[c] = static_cast<uint16_t>(rowbuf_offset(j));
    else
      record_status(a.status, CLQ_ERR_DEVICE_INDEX);
  }
  __syncthreads();

  const int items = R * segs;
  const bool active = tid < items;
  const int r_local = active ? tid / segs : 0;
  const int seg = active ? tid - r_local * segs : 0;
  const int cpr = K >> 3;  // 16-byte chunks per row
  const int total_chunks = R * cpr;
  const int ntiles = (a.M + R - 1) / R;
  const char* Xb = static_cast<const char*>(a.X);
  const size_t ld_bytes = static_cast<size_t>(a.ld) * 2u;

  int par = 0;
  for (int tile = blockIdx.x; tile < ntiles; tile += gridDim.x, par ^= 1) {
    const int row0 = tile * R;

    // ---- phase 1: coalesced loads, scatter to permuted positions ----------
    for (int base = tid; base < total_chunks; base += 4 * nthr) {
      uint4 v[4];
      int rr[4], cc[4];
      bool ok[4];
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const int id = base + u * nthr;
        rr[u] = id / cpr;
        cc[u] = id - rr[u] * cpr;
        ok[u] = id < total_chunks && row0 + rr[u] < a.M;
        if (ok[u])
          v[u] = ld_stream_v4(Xb + static_cast<size_t>(row0 + rr[u]) * ld_bytes +
                              static_cast<size_t>(cc[u]) * 16u);
      }
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        if (!ok[u]) continue;
        const uint4 off = *reinterpret_cast<const uint4*>(dst_off + cc[u] * 8);
        uint8_t* rb = rowbuf + static_cast<size_t>(rr[u]) * 2 * K;
        const uint32_t o[4] = {off.x, off.y, off.z, off.w};
        const uint32_t d[4] = {v[u].x, v[u].y, v[u].z, v[u].w};
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          *reinterpret_cast<uint16_t*>(rb + (o[i] & 0xFFFFu)) =
              static_cast<uint16_t>(d[i] & 0xFFFFu);
          *reinterpret_cast<uint16_t*>(rb + (o[i] >> 16)) =
              static_cast<uint16_t>(d[i] >> 16);
        }
      }
    }
    __syncthreads();

    // ---- phase 2: block Walsh-Hadamard transform and row abs-max ----------
    float v[32];
    {
      const uint8_t* rb = rowbuf + static_cast<size_t>(r_local) * 2 * K;
#pragma unroll
      for (int c = 0; c < 4; ++c) {
        const uint32_t q = static_cast<uint32_t>(seg * 4 + c);
        const uint32_t phys = q ^ ((q >> 3) & 3u);
        const uint4 raw = *reinterpret_cast<const uint4*>(rb + (phys << 4));
        unpack8<T>(raw, v + 8 * c);
      }
    }
    // in-register stages: strides 1 .. min(b, 32) / 2
#pragma unroll
    for (int h = 1; h < 32; h <<= 1) {
      if (h < (1 << LOGB)) {
#pragma unroll
        for (int e = 0; e < 32; ++e) {
          if ((e & h) == 0) {
            const float x0 = v[e], x1 = v[e + h];
            v[e] = x0 + x1;
            v[e + h] = x0 - x1;
          }
        }
      }
    }
    // cross-lane stages: strides 32 .. b / 2, partner lane = lane ^ hl
#pragma unroll
    for (int hl = 1; hl < 8; hl <<= 1) {
      if (LOGB > 5 && hl < (1 << (LOGB > 5 ? LOGB - 5 : 0))) {
        const bool upper = (lane & hl) != 0;
#pragma unroll
        for (int e = 0; e < 32; ++e) {
          const float p = __shfl_xor_sync(0xffffffffu, v[e], hl);
          v[e] = upper ? (p - v[e]) : (v[e] + p);
        }
      }
    }
    float m = 0.f;
#pragma unroll
    for (int e = 0; e < 32; ++e) m = fmaxf(m, fabsf(v[e]));
    {
      // Padding lanes (tid >= items) only keep the shuffles convergent; their
      // values are not data of any row and must not reach a row maximum.
      const int key = active ? r_local : -1;
      const unsigned grp = __match_any_sync(0xffffffffu, key);
      const unsigned mx = __reduce_max_sync(grp, __float_as_uint(m));
      if (active && lane == __ffs(grp) - 1) atomicMax(&amax_s[par * R + r_local], mx);
    }
    __syncthreads();

    // ---- phase 3: scale, codes, pack, store --------------------------------
    const int row = row0 + r_local;
    if (active && row < a.M) {
      float amax = __uint_as_float(amax_s[par * R + r_local]);
      if (a.clip != nullptr) amax = fminf(amax, __ldg(a.clip + row));
      const float s = __fdiv_rn(amax, 7.0f);
      uint32_t w[4] = {0u, 0u, 0u, 0u};
      if (s > 0.f) {
        const float rcp = __frcp_rn(s);
#pragma unroll
        for (int e = 0; e < 32; ++e) {
          const int q = quant_code(v[e], s, rcp);
          w[e >> 3] |= (static_cast<uint32_t>(q) & 0xFu) << (4 * (e & 7));
        }
      }
      uint8_t* qrow = a.Q + static_cast<size_t>(row) * (K >> 1);
      *reinterpret_cast<uint4*>(qrow + seg * 16) = make_uint4(w[0], w[1], w[2], w[3]);
      if (seg == 0) a.S[row] = s;
      if (a.rot != nullptr) {
        float4* dst = reinterpret_cast<float4*>(a.rot + static_cast<size_t>(row) * K + seg * 32);
#pragma unroll
        for (int i = 0; i < 8; ++i)
          dst[i] = make_float4(v[4 * i], v[4 * i + 1], v[4 * i + 2], v[4 * i + 3]);
      }
    }
    if (tid < R) amax_s[(par ^ 1) * R + tid] = 0u;
  }
}

// Outlier score (Sec. 3.3): S = fp32 batch mean (sequential sum over the
// batch, then / B), score[k] = max_t |S[t][k]|.  Threads own channels;
// blockIdx.y owns a slice of tokens; slices combine with an integer atomicMax
// on the (non-negative) float bits, so `scores` must be zeroed first.
template <typename T>
__global__ void outlier_scores_kernel(const uint16_t* calib, int B, int Tn, int K,
                                      int tokens_per_slice, float* scores) {
  const int k = blockIdx.x * blockDim.x + threadIdx.x;
  if (k >= K) return;
  const int t0 = blockIdx.y * tokens_per_slice;
  const int t1 = min(Tn, t0 + tokens_per_slice);
  const size_t bstride = static_cast<size_t>(Tn) * K;
  const float fb = static_cast<float>(B);
  float best = 0.f;
  for (int t = t0; t < t1; ++t) {
    float sum = 0.f;
    for (int b = 0; b < B; ++b)
      sum = sum + Num<T>::to_f(calib[b * bstride + static_cast<size_t>(t) * K + k]);
    best = fmaxf(best, fabsf(__fdiv_rn(sum, fb)));
  }
  atomicMax(reinterpret_cast<unsigned*>(scores) + k, __float_as_uint(best));
}

template <typename T, int LOGB>
cudaError_t launch_rq_t(const RotateQuantArgs& a, int threads, size_t smem, int grid,
                        cudaStream_t st) {
  auto kern = rotate_quant_kernel<T, LOGB>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(smem));
  if (e != cudaSuccess) return e;
  int per_sm = 0;
  e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, threads, smem);
  if (e != cudaSuccess) return e;
  if (per_sm < 1) return cudaErrorInvalidConfiguration;
  const int ntiles = (a.M + a.rows_per_tile - 1) / a.rows_per_tile;
  const int g = std::min(ntiles, grid * per_sm);
  kern<<<g, threads, smem, st>>>(a);
  return cudaGetLastError();
}

template <typename T>
cudaError_t launch_rq_dtype(const RotateQuantArgs& a, int logb, int threads, size_t smem,
                            int grid, cudaStream_t st) {
  switch (logb) {
    case 0: return launch_rq_t<T, 0>(a, threads, smem, grid, st);
    case 1: return launch_rq_t<T, 1>(a, threads, smem, grid, st);
    case 2: return launch_rq_t<T, 2>(a, threads, smem, grid, st);
    case 3: return launch_rq_t<T, 3>(a, threads, smem, grid, st);
    case 4: return launch_rq_t<T, 4>(a, threads, smem, grid, st);
    case 5: return launch_rq_t<T, 5>(a, threads, smem, grid, st);
    case 6: return launch_rq_t<T, 6>(a, threads, smem, grid, st);
    case 7: return launch_rq_t<T, 7>(a, threads, smem, grid, st);
    case 8: return launch_rq_t<T, 8>(a, threads, smem, grid, st);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace

// Rows per tile: the CTA gets one thread per 32-element segment of each of
// its rows.  Prefer thread counts that fill whole warps (padding lanes do no
// useful work) and lie in [192, 384], which keeps two to three CTAs per SM.
void rotate_quant_config(int K, int* rows_per_tile, int* threads, size_t* smem) {
  const int segs = K >> 5;
  int best_r = 1;
  double best_score = -1.0;
  for (int r = 1; r * segs <= 512; ++r) {
    const int t = r * segs;
    const int t32 = (t + 31) & ~31;
    const double fill = static_cast<double>(t) / t32;
    const double size_term =
        t32 < 192 ? t32 / 384.0 : (t32 <= 384 ? 1.0 + t32 / 4096.0 : 0.5);
    const double score = fill * 4.0 + size_term;
    if (score > best_score + 1e-9) {
      best_score = score;
      best_r = r;
    }
  }
  *rows_per_tile = best_r;
  *threads = ((best_r * segs) + 31) & ~31;
  *smem = static_cast<size_t>((2 * K + 15) & ~15) + static_cast<size_t>(best_r) * 2 * K +
          8u * best_r;
}

cudaError_t launch_rotate_quant(const RotateQuantArgs& a, int dtype, int logb,
                                cudaStream_t st) {
  RotateQuantArgs args = a;
  int threads = 0;
  size_t smem = 0;
  rotate_quant_config(a.K, &args.rows_per_tile, &threads, &smem);
  int dev = 0, sms = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  if (e != cudaSuccess) return e;
  if (dtype == CLQ_F16) return launch_rq_dtype<__half>(args, logb, threads, smem, sms, st);
  return launch_rq_dtype<__nv_bfloat16>(args, logb, threads, smem, sms, st);
}

cudaError_t launch_outlier_scores(const void* calib, int dtype, int B, int T, int K,
                                  float* scores, cudaStream_t st) {
  cudaError_t e = cudaMemsetAsync(scores, 0, sizeof(float) * static_cast<size_t>(K), st);
  if (e != cudaSuccess) return e;
  const int threads = 256;
  const int gx = (K + threads - 1) / threads;
  const int slices = std::max(1, std::min(T, 4096 / std::max(gx, 1)));
  const int per = (T + slices - 1) / slices;
  const dim3 grid(gx, (T + per - 1) / per);
  const uint16_t* c = static_cast<const uint16_t*>(calib);
  if (dtype == CLQ_F16)
    outlier_scores_kernel<__half><<<grid, threads, 0, st>>>(c, B, T, K, per, scores);
  else
    outlier_scores_kernel<__nv_bfloat16><<<grid, threads, 0, st>>>(c, B, T, K, per, scores);
  return cudaGetLastError();
}

}  // namespace clq
