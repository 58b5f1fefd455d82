// Fused W4A4 OBS linear: rotate-quant and the tcgen05 GEMM in one persistent
// kernel.
//
// Why not a per-tile prologue: quantizing a token needs the abs-max of its
// whole rotated row before any code exists, and a K step of the product
// needs permuted positions whose source columns are spread over the whole
// row.  For the paper's hidden sizes a 128-token block of rows does not fit
// in shared memory next to the operand pipeline, so each CTA cannot rotate
// only "its" A tile.  Instead rotate-quant (rq::run) writes the codes of
// token rows claimed from a grid-wide counter into the caller's workspace
// and publishes, per 128-token block, how many rows are done; the GEMM
// pipeline (gemm::pipeline) takes the codes in E4M3, so that TMA loads them
// straight into the MMA operand layout, and its TMA producer waits (acquire,
// bounded) until all rows of a tile's token block are published before
// loading that block's codes.  One launch, no host round trip, and the codes
// stay in L2 for the layer sizes of the paper's models.  Rows are claimed,
// not assigned, and rotate-quant never waits on the GEMM, so the producer's
// waits end as long as any CTA runs.
//
// Sequential form (fused_linear_kernel): every CTA first runs rotate-quant
// with all its threads (publishing each tile: proxy fence, CTA barrier,
// __threadfence, atomicAdd), then turns into a GEMM pipeline.
//
// Concurrent form (fused_concurrent_kernel; E4M3 weights, K <= 9216): the
// two run side by side.  Warps 0-5 of every CTA are the GEMM pipeline with
// four epilogue warps and three stages; warps 6-14 rotate and quantize token
// rows in the shared memory the GEMM leaves free, and warp 15 claims their
// tiles, loads and publishes them (rq::run's loader mode).  The GEMM of a
// token block starts as soon as its rows are published.
#include <type_traits>

#include "gemm_pipeline.cuh"
#include "rq_device.cuh"

namespace clq {

namespace {

using namespace gemm;

// Threads per CTA.  Sequential form: rotate-quant on all of them, then the
// GEMM pipeline on up to 448.  Concurrent form: GEMM warps 0-5 beside
// rotate-quant warps 6-15.
constexpr int FT = 512;

// Adds the rows [row0, row0 + rows) to the ready counters of the 128-token
// blocks they fall in (a tile of rows may straddle two blocks); RELEASE: each
// add is a release at GPU scope, else relaxed (the caller fences first).
template <bool RELEASE>
__device__ __forceinline__ void count_rows(uint32_t* ready, int row0, int rows) {
  int r = row0;
  const int end = row0 + rows;
  while (r < end) {
    const int mb = r / BM;
    const int stop = min(end, (mb + 1) * BM);
    const unsigned n = static_cast<unsigned>(stop - r);
    if (RELEASE)
      asm volatile("red.release.gpu.global.add.u32 [%0], %1;" ::"l"(ready + mb), "r"(n)
                   : "memory");
    else
      atomicAdd(ready + mb, n);
    r = stop;
  }
}

struct PublishRows {
  uint32_t* ready;
  rq::Team team;  // the threads that stored the rows
  // Every team thread, once its stores of the tile are issued: proxy fence,
  // team barrier, then one thread publishes (fence at GPU scope, adds).
  __device__ void operator()(int row0, int rows) const {
    fence_proxy_async_global();
    team.sync();
    if (team.rank() == 0) {
      __threadfence();
      count_rows<false>(ready, row0, rows);
    }
  }
  // Loader mode: the compute threads have fenced their stores for the async
  // proxy and signalled them on a CTA barrier this thread has waited on; a
  // release add at GPU scope makes them visible to every CTA that acquires
  // the counter.
  __device__ void release(int row0, int rows) const { count_rows<true>(ready, row0, rows); }
};

// Rotate-quant stage geometry of the fused kernel: its shared memory is sized
// for the GEMM pipeline anyway, so 32 KB stages let 512 threads cover as many
// rows per tile as they can (14 rows at K = 1152, 3 at K = 4608).
constexpr int kRqStride = 32 * 1024;
constexpr int kRqStages = 4;

// Concurrent form: GEMM warps 0-5, rotate-quant team warps 6-15 (compute
// warps 6-14, loader warp 15).
constexpr int kTeamFirst = (WARP_MMA + 1) * 32;  // 192
constexpr int kTeamThreads = FT - kTeamFirst;     // 320
constexpr int kTeamCompute = kTeamThreads - 32;   // 288
constexpr uint32_t kTeamBarrier = 2;  // 0: CTA, 1: GEMM epilogue, 2-3: team
constexpr int kConcStride = 19 * 1024;
constexpr int kConcStages = 3;
constexpr int kConcGemmStages = 3;

template <int BNT>
struct Conc {
  using C = Cfg<false, false, BNT, 1, 1, 4, kConcGemmStages>;
  static constexpr size_t RQ_OFF = (C::BYTES + 1023) & ~static_cast<size_t>(1023);
};

// F6 (both forms): the workspace codes and the weights are E2M3, loaded by
// 16U6 tensor maps (gemm::pipeline's F6 mode).
template <typename T, bool BPACK, int BNT, bool F6>
__global__ void __launch_bounds__(FT, 1)
    fused_linear_kernel(const __grid_constant__ CUtensorMap mapA,
                        const __grid_constant__ CUtensorMap mapB,
                        const __grid_constant__ CUtensorMap mapY, RotateQuantArgs rq, GemmArgs g,
                        uint32_t* ready, uint32_t* tile_counter, int use_tma_store) {
  extern __shared__ uint8_t smem_raw[];
  __shared__ Barriers bars;
  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  setup<false, BPACK, BNT>(&bars);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = bars.tmem_slot;

  rq::run<T, -1, false, kRqStride, kRqStages>(rq, smem, tile_counter,
                                              PublishRows{ready, rq::Team()});
  __syncthreads();

  const Maps maps{&mapA, &mapB, use_tma_store ? &mapY : nullptr};
  pipeline<T, false, BPACK, BNT, false, 1, 1, false, 0, MAX_STAGES, F6>(maps, g, smem, &bars,
                                                                        tmem, ready);
  tc_fence_before();
  __syncthreads();
  teardown(tmem, Cfg<false, BPACK, BNT>::TMEM);
}

template <typename T, int BNT, bool F6>
__global__ void __launch_bounds__(FT, 1)
    fused_concurrent_kernel(const __grid_constant__ CUtensorMap mapA,
                            const __grid_constant__ CUtensorMap mapB,
                            const __grid_constant__ CUtensorMap mapY, RotateQuantArgs rq,
                            GemmArgs g, uint32_t* ready, uint32_t* tile_counter,
                            int use_tma_store) {
  using C = typename Conc<BNT>::C;
  extern __shared__ uint8_t smem_raw[];
  __shared__ Barriers bars;
  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  setup<false, false, BNT, 1, 1, 4, kConcGemmStages>(&bars);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = bars.tmem_slot;

  if (static_cast<int>(threadIdx.x) >= kTeamFirst) {
    rq::Team team;
    team.first = kTeamFirst;
    team.count = kTeamThreads;
    team.bar = kTeamBarrier;
    rq::run<T, -1, false, kConcStride, kConcStages, false, false, PublishRows, true>(
        rq, smem + Conc<BNT>::RQ_OFF, tile_counter, PublishRows{ready, team}, team);
  } else {
    const Maps maps{&mapA, &mapB, use_tma_store ? &mapY : nullptr, nullptr, nullptr};
    pipeline<T, false, false, BNT, false, 1, 1, false, 4, kConcGemmStages, F6>(maps, g, smem,
                                                                              &bars, tmem, ready);
  }
  tc_fence_before();
  __syncthreads();
  teardown(tmem, C::TMEM);
}

template <typename T, int BNT, bool F6>
cudaError_t launch_conc(const CUtensorMap& mapA, const CUtensorMap& mapB,
                        const CUtensorMap& mapY, const RotateQuantArgs& rq, const GemmArgs& g,
                        uint32_t* ready, int use_tma_store, size_t smem, int grid,
                        cudaStream_t st) {
  uint32_t* tile_counter = ready + (g.M + BM - 1) / BM;
  auto k = fused_concurrent_kernel<T, BNT, F6>;
  cudaError_t e = kernel_setup(reinterpret_cast<const void*>(k), smem, FT, nullptr);
  if (e != cudaSuccess) return e;
  k<<<grid, FT, smem, st>>>(mapA, mapB, mapY, rq, g, ready, tile_counter, use_tma_store);
  return cudaGetLastError();
}

template <typename T, bool BPACK, int BNT, bool F6>
cudaError_t launch_t(const CUtensorMap& mapA, const CUtensorMap& mapB, const CUtensorMap& mapY,
                     const RotateQuantArgs& rq, const GemmArgs& g, uint32_t* ready,
                     int use_tma_store, size_t smem, int grid, cudaStream_t st) {
  uint32_t* tile_counter = ready + (g.M + BM - 1) / BM;
  auto k = fused_linear_kernel<T, BPACK, BNT, F6>;
  cudaError_t e = kernel_setup(reinterpret_cast<const void*>(k), smem, FT, nullptr);
  if (e != cudaSuccess) return e;
  k<<<grid, FT, smem, st>>>(mapA, mapB, mapY, rq, g, ready, tile_counter, use_tma_store);
  return cudaGetLastError();
}


size_t align256(size_t x) { return (x + 255) & ~static_cast<size_t>(255); }

}  // namespace

FusedWorkspace fused_workspace_layout(int M, int K) {
  FusedWorkspace w{};
  const size_t m = static_cast<size_t>(M < 0 ? 0 : M);
  w.codes_off = 0;
  w.scales_off = align256(m * static_cast<size_t>(K));  // E4M3 codes
  w.ready_off = align256(w.scales_off + 4 * m);
  w.bytes = align256(w.ready_off + 4 * ((m + BM - 1) / BM + 1));  // + tile counter
  return w;
}

namespace {

// Concurrent form (E4M3 weights): rows per tile as the 288 compute threads
// and a 19 KB stage allow (8 at K = 1152, 2 at K = 4608).
cudaError_t launch_concurrent(const RotateQuantArgs& rq_in, const uint8_t* W, int w_codes,
                              const GemmArgs& g, int logb, int dtype, uint32_t* ready, int sms,
                              cudaStream_t st) {
  RotateQuantArgs rq = rq_in;
  rq.logb = logb;
  const bool f6 = w_codes == CLQ_CODES_E2M3;
  const int a_codes = f6 ? CLQ_CODES_E2M3 : CLQ_CODES_E4M3;  // the weights' family
  rq.e4m3 = f6 ? 3 : 1;
  const int segs = rq.K / 32;
  const int R = std::min(kTeamCompute / segs, kConcStride / (2 * rq.K));
  if (R < 1) return cudaErrorInvalidValue;
  rq.rows_per_tile = R;
  const int bn = gemm_tile_n(g.M, g.N, sms);
  const size_t gemm_off = bn == 192 ? Conc<192>::RQ_OFF : Conc<256>::RQ_OFF;
  const size_t smem = gemm_off + rq::smem_bytes(R, kConcStride, kConcStages) + 1024;
  if (smem > 227u * 1024u - 2048u) return cudaErrorInvalidValue;

  const int tiles_m = (g.M + BM - 1) / BM;
  cudaError_t e =
      cudaMemsetAsync(ready, 0, sizeof(uint32_t) * (static_cast<size_t>(tiles_m) + 1), st);
  if (e != cudaSuccess) return e;
  CUtensorMap mapA, mapB, mapY;
  if (!encode_codes_map(&mapA, rq.Q, a_codes, g.M, g.K, BM, 0) ||
      !encode_codes_map(&mapB, W, w_codes, g.N, g.K, bn, 0))
    return cudaErrorInvalidValue;
  const int use_tma_store = (g.N % 8 == 0) ? 1 : 0;
  if (use_tma_store) {
    if (!encode_tma_out_tile(&mapY, g.Y, g.M, g.N)) return cudaErrorInvalidValue;
  } else {
    mapY = mapA;  // unused
  }
  auto go = [&](auto f6_tag) {
    constexpr bool F6 = decltype(f6_tag)::value;
    if (dtype == CLQ_F16)
      return bn == 192 ? launch_conc<__half, 192, F6>(mapA, mapB, mapY, rq, g, ready,
                                                      use_tma_store, smem, sms, st)
                       : launch_conc<__half, 256, F6>(mapA, mapB, mapY, rq, g, ready,
                                                      use_tma_store, smem, sms, st);
    return bn == 192 ? launch_conc<__nv_bfloat16, 192, F6>(mapA, mapB, mapY, rq, g, ready,
                                                           use_tma_store, smem, sms, st)
                     : launch_conc<__nv_bfloat16, 256, F6>(mapA, mapB, mapY, rq, g, ready,
                                                           use_tma_store, smem, sms, st);
  };
  return f6 ? go(std::true_type()) : go(std::false_type());
}

}  // namespace

cudaError_t launch_fused_linear(const RotateQuantArgs& rq_in, const uint8_t* W, int w_codes,
                                const GemmArgs& g, int logb, int dtype, uint32_t* ready,
                                cudaStream_t st) {
  const bool bpack = w_codes == CLQ_CODES_INT4_PACKED;
  const int sms = sm_count();
  if (sms <= 0) return cudaErrorInvalidDevice;
  if (!bpack && rq_in.K <= kConcStride / 2 && rq_in.K / 32 <= kTeamCompute)
    return launch_concurrent(rq_in, W, w_codes, g, logb, dtype, ready, sms, st);
  const int bn = BN;
  const size_t gemm_bytes = bpack ? Cfg<false, true>::BYTES : Cfg<false, false>::BYTES;
  const size_t limit = 227u * 1024u - 2048u;  // dynamic + static shared memory
  // Rotate-quant phase: as many rows per tile as 512 threads cover and one
  // raw stage holds.
  RotateQuantArgs rq = rq_in;
  rq.logb = logb;
  // the workspace holds the codes in the GEMM's operand layout: E2M3 beside
  // E2M3 weights, else E4M3
  const bool f6 = w_codes == CLQ_CODES_E2M3;
  rq.e4m3 = f6 ? 3 : 1;
  const int segs = rq.K / 32;
  const int R = std::max(1, std::min(FT / segs, kRqStride / (2 * rq.K)));
  const size_t rq_bytes = rq::smem_bytes(R, kRqStride, kRqStages);
  if (rq_bytes > limit || R * segs > FT) return cudaErrorInvalidValue;
  rq.rows_per_tile = R;
  const size_t smem = std::max(gemm_bytes, rq_bytes) + 1024;

  const int tiles_m = (g.M + BM - 1) / BM;
  cudaError_t e =
      cudaMemsetAsync(ready, 0, sizeof(uint32_t) * (static_cast<size_t>(tiles_m) + 1), st);
  if (e != cudaSuccess) return e;

  CUtensorMap mapA, mapB, mapY;
  if (!encode_codes_map(&mapA, rq.Q, f6 ? CLQ_CODES_E2M3 : CLQ_CODES_E4M3, g.M, g.K, BM, 0) ||
      !encode_codes_map(&mapB, W, w_codes, g.N, g.K, bn, 0))
    return cudaErrorInvalidValue;
  const int use_tma_store = (g.N % 8 == 0) ? 1 : 0;
  if (use_tma_store) {
    if (!encode_tma_out_tile(&mapY, g.Y, g.M, g.N)) return cudaErrorInvalidValue;
  } else {
    mapY = mapA;  // unused
  }
  const int grid = sms;
  if (f6)
    return dtype == CLQ_F16
               ? launch_t<__half, false, BN, true>(mapA, mapB, mapY, rq, g, ready, use_tma_store,
                                                   smem, grid, st)
               : launch_t<__nv_bfloat16, false, BN, true>(mapA, mapB, mapY, rq, g, ready,
                                                          use_tma_store, smem, grid, st);
  if (dtype == CLQ_F16)
    return bpack ? launch_t<__half, true, BN, false>(mapA, mapB, mapY, rq, g, ready,
                                                     use_tma_store, smem, grid, st)
                 : launch_t<__half, false, BN, false>(mapA, mapB, mapY, rq, g, ready,
                                                      use_tma_store, smem, grid, st);
  return bpack ? launch_t<__nv_bfloat16, true, BN, false>(mapA, mapB, mapY, rq, g, ready,
                                                          use_tma_store, smem, grid, st)
               : launch_t<__nv_bfloat16, false, BN, false>(mapA, mapB, mapY, rq, g, ready,
                                                           use_tma_store, smem, grid, st);
}

}  // namespace clq
