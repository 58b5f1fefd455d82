// Rotate-quantize launch configuration and dispatch (the kernels are in
// rotate_quant_f16.cu / rotate_quant_bf16.cu, the tile loop in
// rq_device.cuh) and the outlier-score kernel.
#include "rq_launch.cuh"

namespace clq {

namespace {

// Cost-model constants of the paired kernel (us, elements per us per SM).
constexpr double kPairFloorUs = 1.0;
constexpr double kPairRate = 10000.0;
constexpr double kPairFirstUs = 0.25;

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

}  // namespace

// Rows per tile: the CTA gets one thread per 32-element segment of each of
// its rows, R rows fitting one raw stage (2 R K bytes).  At 128 registers a
// thread an SM holds 16 warps.  R is chosen by a cost model fitted to timings
// on GB300 (M up to 65536 tokens): a CTA takes about max(1.2, 0.1 + 0.121 W)
// us per tile when W warps share the SM (a latency floor, then issue-bound),
// every CTA walks ceil(tiles / CTAs) tiles, and the first tile's arrival adds
// about 0.25 us per 2304-byte row (refit after the XOR-ordered gather: a sweep
// of rows per tile over the benchmark shapes); a lone CTA per SM pays 1.35x
// per tile.  Few
// rows per tile win when M is small (more CTAs share the work), many when M
// is large.
void rotate_quant_config(int M, int K, int sms, int* rows_per_tile, int* threads,
                         size_t* smem) {
  const int segs = K >> 5;
  const int stride = rq::kStride;
  const int stages = rq::kStages;
  int best_r = 1;
  double best_cost = 1e300;
  for (int r = 1; r * segs <= 512 && 2 * r * K <= stride; ++r) {
    const int warps = (r * segs + 31) / 32;
    const size_t bytes = rq::smem_bytes(r, stride, stages);
    const int by_warps = (65536 / (32 * rq::kMaxRegs)) / warps;
    const int by_smem = static_cast<int>((227u * 1024u) / (bytes + 1024u));
    const int ctas = std::min(by_warps, by_smem);
    if (ctas < 1) continue;
    const long tiles = (static_cast<long>(M) + r - 1) / r;
    const long total = static_cast<long>(ctas) * std::max(sms, 1);
    const long rounds = (tiles + total - 1) / total;
    // A lone CTA per SM has no second CTA to run through its barrier stalls
    // (measured: 1.35x per tile at K = 4608).
    const double alone = ctas == 1 ? 1.35 : 1.0;
    const double cost = rounds * alone * std::max(1.2, 0.1 + 0.121 * ctas * warps) +
                        0.25 * r * (2.0 * K) / 2304.0;
    if (cost < best_cost - 1e-9) {
      best_cost = cost;
      best_r = r;
    }
  }
  *rows_per_tile = best_r;
  *threads = ((best_r * segs) + 31) & ~31;
  *smem = rq::smem_bytes(best_r, stride, stages);
}

// Paired-row kernel (rq_pair.cuh): RH rows per half-stage, chosen by the same
// kind of model: an SM runs a round of its resident CTAs' tiles in about
// max(floor, elements / (rate * min(1, warps / 16))) us (issue-bound with
// enough warps, latency-bound below; 16 warps a SM measured 8 % faster than
// 12 at 16384 x 1152, b = 128), the CTAs walk ceil(tiles / CTAs) rounds, and
// the first tile's arrival adds its bytes' share of latency.
void rotate_quant_pair_config(int M, int K, int sms, int* rows_half, int* threads, size_t* smem,
                              int* half) {
  const int row = 2 * K;
  const int hb = row <= rq::kPairHalfSmall ? rq::kPairHalfSmall : rq::kPairHalfLarge;
  const int segs = K >> 5;
  const int rh_max = std::max(1, std::min(hb / row, 512 / segs));
  const int regs_warps = 65536 / (32 * rq::kPairMaxRegs);
  int best = 1;
  double best_cost = 1e300;
  for (int rh = 1; rh <= rh_max; ++rh) {
    const int warps = (rh * segs + 31) / 32;
    const size_t bytes = rq::pair_smem_bytes(rh, hb, rq::kPairStages);
    const int ctas = std::min(regs_warps / warps, static_cast<int>((227u * 1024u) / (bytes + 1024u)));
    if (ctas < 1) continue;
    const long tiles = (static_cast<long>(M) + 2 * rh - 1) / (2 * rh);
    const long total = static_cast<long>(ctas) * std::max(sms, 1);
    const long rounds = (tiles + total - 1) / total;
    const double elems = static_cast<double>(ctas) * 2 * rh * K;
    const double occ = std::min(1.0, ctas * warps / 16.0);
    const double round_us = std::max(kPairFloorUs, elems / (kPairRate * occ));
    const double cost = rounds * round_us + kPairFirstUs * (2.0 * rh * row) / 4608.0;
    if (cost < best_cost - 1e-9) {
      best_cost = cost;
      best = rh;
    }
  }
  *rows_half = best;
  *threads = ((best * segs) + 31) & ~31;
  *smem = rq::pair_smem_bytes(best, hb, rq::kPairStages);
  *half = hb;
}

// Wide-segment kernel (rq_wide.cuh): RH rows a tile, one thread per 64
// positions of a row, stage STAGE bytes; the same model as the paired
// kernel with the register cap of the wide loop.
void rotate_quant_wide_config(int M, int K, int sms, int* rows, int* threads, size_t* smem,
                              int* stage) {
  const int row = 2 * K;
  const int sb = row <= rq::kPairHalfSmall ? rq::kPairHalfSmall : rq::kPairHalfLarge;
  const int segs = K >> 6;
  const int rh_max = std::max(1, std::min(sb / row, 512 / segs));
  const int regs_warps = 65536 / (32 * rq::kWideMaxRegs);
  int best = 1;
  double best_cost = 1e300;
  for (int rh = 1; rh <= rh_max; ++rh) {
    const int warps = (rh * segs + 31) / 32;
    const size_t bytes = rq::wide_smem_bytes(rh, sb, rq::kPairStages);
    const int ctas = std::min(regs_warps / warps, static_cast<int>((227u * 1024u) / (bytes + 1024u)));
    if (ctas < 1) continue;
    const long tiles = (static_cast<long>(M) + rh - 1) / rh;
    const long total = static_cast<long>(ctas) * std::max(sms, 1);
    const long rounds = (tiles + total - 1) / total;
    // idle lanes of a partial last warp cost like working ones
    const double elems = static_cast<double>(ctas) * warps * 32 * 64;
    const double occ = std::min(1.0, ctas * warps / 12.0);
    const double round_us = std::max(kPairFloorUs, elems / (kPairRate * occ));
    const double cost = rounds * round_us + kPairFirstUs * (rh * row) / 4608.0;
    if (cost < best_cost - 1e-9) {
      best_cost = cost;
      best = rh;
    }
  }
  *rows = best;
  *threads = ((best * segs) + 31) & ~31;
  *smem = rq::wide_smem_bytes(best, sb, rq::kPairStages);
  *stage = sb;
}

cudaError_t launch_rotate_quant(const RotateQuantArgs& a, int dtype, int logb,
                                cudaStream_t st) {
  RotateQuantArgs args = a;
  int threads = 0;
  size_t smem = 0;
  const int sms = sm_count();
  if (sms <= 0) return cudaErrorInvalidDevice;
  // Symmetric 4-bit activation codes in the E4M3 or E2M3 layout: the wide
  // kernel for b = 64 (K % 64 == 0; measured 10 % faster in the PixArt step
  // than the paired kernel, which wins at b = 128 and 256), the paired-row
  // kernel for 32 <= b <= 256 otherwise.
  const bool hot = a.lo == nullptr && a.clip == nullptr && (a.e4m3 == 1 || a.e4m3 == 3);
  // Asymmetric 4-bit codes in E4M3 bytes take the wide kernel too (b = 64).
  const bool hot_asym = a.lo != nullptr && a.clip == nullptr && a.e4m3 == 1;
  if ((hot || hot_asym) && logb == 6 && a.K % 64 == 0) {
    int stage = 0;
    rotate_quant_wide_config(a.M, a.K, sms, &args.rows_per_tile, &threads, &smem, &stage);
    const bool e2 = a.e4m3 == 3;
    if (dtype == CLQ_F16)
      return e2 ? launch_rotate_quant_wide_f16_e2m3(args, logb, stage, threads, smem, sms, st)
                : launch_rotate_quant_wide_f16_e4m3(args, logb, stage, threads, smem, sms, st);
    return e2 ? launch_rotate_quant_wide_bf16_e2m3(args, logb, stage, threads, smem, sms, st)
              : launch_rotate_quant_wide_bf16_e4m3(args, logb, stage, threads, smem, sms, st);
  }
  if (hot && logb >= 5) {
    int half = 0;
    rotate_quant_pair_config(a.M, a.K, sms, &args.rows_per_tile, &threads, &smem, &half);
    const bool e2 = a.e4m3 == 3;
    if (dtype == CLQ_F16)
      return e2 ? launch_rotate_quant_pair_f16_e2m3(args, logb, half, threads, smem, sms, st)
                : launch_rotate_quant_pair_f16_e4m3(args, logb, half, threads, smem, sms, st);
    return e2 ? launch_rotate_quant_pair_bf16_e2m3(args, logb, half, threads, smem, sms, st)
              : launch_rotate_quant_pair_bf16_e4m3(args, logb, half, threads, smem, sms, st);
  }
  rotate_quant_config(a.M, a.K, sms, &args.rows_per_tile, &threads, &smem);
  if (dtype == CLQ_F16) return launch_rotate_quant_f16(args, logb, threads, smem, sms, st);
  return launch_rotate_quant_bf16(args, logb, threads, smem, sms, st);
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
