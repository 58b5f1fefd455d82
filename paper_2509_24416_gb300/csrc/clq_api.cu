// C ABI of libclq (declared in include/clq.h): argument validation, the host
// column-swap builder, the device status word and kernel launches.  Nothing
// here allocates device memory or synchronizes, except
// clq_get_device_status, which synchronizes by design.
#include <algorithm>
#include <atomic>
#include <cmath>
#include <cstdint>
#include <numeric>
#include <vector>

#include <cuda_runtime.h>

#include "../../include/clq.h"
#include "clq_kernels.h"

namespace {

// Device status word: first device-side error since the last read.
__device__ int32_t g_device_status;

constexpr int kMaxDevices = 64;
std::atomic<int32_t*> g_status_ptr[kMaxDevices];
std::atomic<int> g_arch_ok[kMaxDevices];  // 0 unknown, 1 sm_103, -1 other

bool aligned(const void* p, uintptr_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }

bool pow2_le256(int b) { return b >= 1 && b <= 256 && (b & (b - 1)) == 0; }

int log2i(int b) {
  int l = 0;
  while ((1 << l) < b) ++l;
  return l;
}

clq_status from_cuda(cudaError_t e) { return e == cudaSuccess ? CLQ_OK : CLQ_ERR_CUDA; }

// Current device's status-word address and architecture check.  The first
// call on a device resolves the symbol address; later calls read the cache.
clq_status device_setup(int32_t** status) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return CLQ_ERR_CUDA;
  if (dev < 0 || dev >= kMaxDevices) return CLQ_ERR_UNSUPPORTED;
  int arch = g_arch_ok[dev].load(std::memory_order_acquire);
  if (arch == 0) {
    int major = 0, minor = 0;
    if (cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev) != cudaSuccess)
      return CLQ_ERR_CUDA;
    arch = (major == 10 && minor == 3) ? 1 : -1;
    g_arch_ok[dev].store(arch, std::memory_order_release);
  }
  if (arch != 1) return CLQ_ERR_UNSUPPORTED;
  int32_t* p = g_status_ptr[dev].load(std::memory_order_acquire);
  if (p == nullptr) {
    void* q = nullptr;
    if (cudaGetSymbolAddress(&q, g_device_status) != cudaSuccess) return CLQ_ERR_CUDA;
    p = static_cast<int32_t*>(q);
    g_status_ptr[dev].store(p, std::memory_order_release);
  }
  *status = p;
  return CLQ_OK;
}

clq_status check_k_b(int K, int b) {
  if (!pow2_le256(b)) return CLQ_ERR_SHAPE;
  if (K < 32 || K > 16384 || K % 32 != 0 || K % b != 0) return CLQ_ERR_SHAPE;
  return CLQ_OK;
}

bool valid_dtype(int d) { return d == CLQ_F16 || d == CLQ_BF16; }

// 4-bit layouts (W4A4 entry points) and every layout (rotate-quant, clq_linear).
bool valid_codes(int f) {
  return f == CLQ_CODES_INT4_PACKED || f == CLQ_CODES_E4M3 || f == CLQ_CODES_E2M3;
}

// Extra rules of the E2M3 layout: whole 128-code groups (the GEMM's tensor
// maps take 128 codes a row per box) and 32-byte aligned arrays.
clq_status check_e2m3(int codes, int K, const void* p) {
  if (codes != CLQ_CODES_E2M3) return CLQ_OK;
  if (K % 128 != 0) return CLQ_ERR_SHAPE;
  if (p != nullptr && (reinterpret_cast<uintptr_t>(p) % 32) != 0) return CLQ_ERR_ALIGN;
  return CLQ_OK;
}
bool valid_any_codes(int f) { return valid_codes(f) || f == CLQ_CODES_E4M3_SPLIT; }

// Launch of the fused kernel on a workspace laid out as `ws` (validated).
clq_status fused_common(const void* X, clq_dtype dtype, int32_t M, int32_t K, int32_t ldx,
                        const int32_t* perm, int32_t b, const uint8_t* W, clq_codes w_codes,
                        const float* s_w, const void* bias, int32_t N, void* Y, uint8_t* wsp,
                        const clq::FusedWorkspace& ws, int32_t* status, void* stream) {
  clq::RotateQuantArgs rq{};
  rq.X = X;
  rq.M = M;
  rq.K = K;
  rq.ld = ldx;
  rq.perm = perm;
  rq.clip = nullptr;
  rq.Q = wsp + ws.codes_off;
  rq.S = reinterpret_cast<float*>(wsp + ws.scales_off);
  rq.rot = nullptr;
  rq.status = status;
  clq::GemmArgs g{};
  g.s_x = rq.S;
  g.s_w = s_w;
  g.bias = bias;
  g.Y = Y;
  g.acc_dbg = nullptr;
  g.M = M;
  g.N = N;
  g.K = K;
  g.inv_b = 1.0f / static_cast<float>(b);
  g.status = status;
  return from_cuda(clq::launch_fused_linear(rq, W, w_codes, g, log2i(b), dtype,
                                            reinterpret_cast<uint32_t*>(wsp + ws.ready_off),
                                            static_cast<cudaStream_t>(stream)));
}

clq_status rotate_quant_common(const void* X, clq_dtype dtype, int32_t M, int32_t K, int32_t ld,
                               const int32_t* perm, int32_t b, const float* clip, int codes,
                               uint8_t* Q, float* S, float* rot, void* stream,
                               float* lo = nullptr, bool weights = false) {
  if (!valid_dtype(dtype) || !valid_any_codes(codes) || M < 0) return CLQ_ERR_INVALID_ARG;
  // centered asymmetric codes reach -8, which E2M3 does not hold
  if (lo != nullptr && codes == CLQ_CODES_E2M3) return CLQ_ERR_UNSUPPORTED;
  clq_status st = check_k_b(K, b);
  if (st != CLQ_OK) return st;
  if (codes == CLQ_CODES_E2M3 && K % 128 != 0) return CLQ_ERR_SHAPE;
  if (ld < K) return CLQ_ERR_SHAPE;
  if (ld % 8 != 0) return CLQ_ERR_ALIGN;
  if (M == 0) return CLQ_OK;
  if (X == nullptr || perm == nullptr || Q == nullptr || S == nullptr) return CLQ_ERR_INVALID_ARG;
  if (!aligned(X, 16) || !aligned(Q, 16) || !aligned(perm, 4) || !aligned(S, 4) ||
      (rot != nullptr && !aligned(rot, 16)) || (clip != nullptr && !aligned(clip, 4)) ||
      (lo != nullptr && !aligned(lo, 4)))
    return CLQ_ERR_ALIGN;
  st = check_e2m3(codes, K, Q);
  if (st != CLQ_OK) return st;
  int32_t* status = nullptr;
  st = device_setup(&status);
  if (st != CLQ_OK) return st;
  clq::RotateQuantArgs a{};
  a.X = X;
  a.M = M;
  a.K = K;
  a.ld = ld;
  a.perm = perm;
  a.clip = clip;
  a.Q = Q;
  a.S = S;
  a.rot = rot;
  a.lo = lo;
  a.status = status;
  a.serial = weights ? 1 : 0;
  a.logb = log2i(b);
  a.e4m3 = codes == CLQ_CODES_E4M3         ? 1
           : codes == CLQ_CODES_E4M3_SPLIT ? 2
           : codes == CLQ_CODES_E2M3       ? 3
                                           : 0;
  return from_cuda(
      clq::launch_rotate_quant(a, dtype, log2i(b), static_cast<cudaStream_t>(stream)));
}

// The product with its epilogue; lo / wsum non-null select the asymmetric
// (zero-point) epilogue.
clq_status linear_common(const uint8_t* Xq, int x_codes, const float* s_x, const float* lo,
                         const uint8_t* W, int w_codes, const float* s_w, const float* wsum,
                         const void* bias, int32_t M, int32_t N, int32_t K, int32_t b,
                         int out_dtype, void* Y, int32_t* acc_dbg, void* stream) {
  if (!valid_dtype(out_dtype) || !valid_any_codes(x_codes) || !valid_any_codes(w_codes) ||
      M < 0 || N < 0)
    return CLQ_ERR_INVALID_ARG;
  // 8-bit operands: W4A8 (split activations, E4M3 weights) and W8A8 only.
  if ((x_codes == CLQ_CODES_E4M3_SPLIT || w_codes == CLQ_CODES_E4M3_SPLIT) &&
      !(x_codes == CLQ_CODES_E4M3_SPLIT &&
        (w_codes == CLQ_CODES_E4M3 || w_codes == CLQ_CODES_E4M3_SPLIT)))
    return CLQ_ERR_UNSUPPORTED;
  // E2M3 operands pair with each other only, symmetric codes only.
  if ((x_codes == CLQ_CODES_E2M3) != (w_codes == CLQ_CODES_E2M3) ||
      (x_codes == CLQ_CODES_E2M3 && lo != nullptr))
    return CLQ_ERR_UNSUPPORTED;
  clq_status st = check_k_b(K, b);
  if (st != CLQ_OK) return st;
  if (x_codes == CLQ_CODES_E2M3 && K % 128 != 0) return CLQ_ERR_SHAPE;
  if (M == 0 || N == 0) return CLQ_OK;
  if (Xq == nullptr || s_x == nullptr || W == nullptr || s_w == nullptr || Y == nullptr)
    return CLQ_ERR_INVALID_ARG;
  if (!aligned(Xq, 16) || !aligned(W, 16) || !aligned(Y, 16) || !aligned(s_x, 4) ||
      !aligned(s_w, 4) || (bias != nullptr && !aligned(bias, 2)) ||
      (acc_dbg != nullptr && !aligned(acc_dbg, 4)) || (lo != nullptr && !aligned(lo, 4)) ||
      (wsum != nullptr && !aligned(wsum, 4)))
    return CLQ_ERR_ALIGN;
  if ((st = check_e2m3(x_codes, K, Xq)) != CLQ_OK || (st = check_e2m3(w_codes, K, W)) != CLQ_OK)
    return st;
  int32_t* status = nullptr;
  st = device_setup(&status);
  if (st != CLQ_OK) return st;
  clq::GemmArgs g{};
  g.s_x = s_x;
  g.s_w = s_w;
  g.bias = bias;
  g.Y = Y;
  g.acc_dbg = acc_dbg;
  g.M = M;
  g.N = N;
  g.K = K;
  g.inv_b = 1.0f / static_cast<float>(b);
  g.status = status;
  g.lo = lo;
  g.wsum = wsum;
  g.zp_shift = x_codes == CLQ_CODES_E4M3_SPLIT ? 128.0f : 8.0f;
  return from_cuda(
      clq::launch_w4a4_gemm(Xq, x_codes, W, w_codes, g, out_dtype,
                            static_cast<cudaStream_t>(stream)));
}

// Workspace of clq_clip_search, 256-byte aligned pieces.
struct ClipWorkspace {
  size_t w_rot, wq, s_w, table, clip, xq, s_x, yh, partial, errors, bytes;
};
constexpr int kClipPartials = 256;

size_t align256(size_t x) { return (x + 255) & ~static_cast<size_t>(255); }

int clip_table_width(int K, const float* grid, int G) {
  int J = 1;
  for (int g = 0; g < G; ++g)
    J = std::max(J, static_cast<int>(std::floor(static_cast<double>(grid[g]) * K)) + 1);
  return J;
}

ClipWorkspace clip_workspace_layout(int M, int N, int K, int J, int G) {
  ClipWorkspace w{};
  size_t off = 0;
  auto take = [&](size_t bytes) {
    const size_t at = off;
    off = align256(off + bytes);
    return at;
  };
  w.w_rot = take(static_cast<size_t>(N) * K * 4);
  w.wq = take(static_cast<size_t>(N) * K);
  w.s_w = take(static_cast<size_t>(N) * 4);
  w.table = take(static_cast<size_t>(N) * J * 4);
  w.clip = take(static_cast<size_t>(N) * 4);
  w.xq = take(static_cast<size_t>(M) * K);
  w.s_x = take(static_cast<size_t>(M) * 4);
  w.yh = take(static_cast<size_t>(M) * N * 2);
  w.partial = take(static_cast<size_t>(G) * kClipPartials * 8);
  w.errors = take(static_cast<size_t>(G) * 8);
  w.bytes = off;
  return w;
}

}  // namespace

namespace clq {
// peaks.cu
cudaError_t launch_peak_rq_stream(const void* X, int M, int K, uint8_t* Q, float* S,
                                  int32_t* status, cudaStream_t st, long long* bytes);
}  // namespace clq

extern "C" {

const char* clq_status_string(clq_status s) {
  switch (s) {
    case CLQ_OK: return "CLQ_OK";
    case CLQ_ERR_INVALID_ARG: return "CLQ_ERR_INVALID_ARG: null pointer, bad enum or negative size";
    case CLQ_ERR_SHAPE: return "CLQ_ERR_SHAPE: shape rule violated (b, K, ld)";
    case CLQ_ERR_ALIGN: return "CLQ_ERR_ALIGN: pointer or stride not aligned";
    case CLQ_ERR_UNSUPPORTED: return "CLQ_ERR_UNSUPPORTED: no sm_103 device or feature";
    case CLQ_ERR_CUDA: return "CLQ_ERR_CUDA: a CUDA runtime call failed";
    case CLQ_ERR_TIMEOUT: return "CLQ_ERR_TIMEOUT: a bounded device-side wait ran out";
    case CLQ_ERR_DEVICE_INDEX: return "CLQ_ERR_DEVICE_INDEX: perm index outside [0, K)";
    case CLQ_ERR_DEVICE_CODE:
      return "CLQ_ERR_DEVICE_CODE: a code array held a value outside [-7, 7]";
    case CLQ_ERR_SCRATCH_LIMIT:
      return "CLQ_ERR_SCRATCH_LIMIT: M x K needs more than the static scratch of "
             "clq_fused_linear_noalloc";
    default: return "unknown clq_status";
  }
}

int32_t clq_version(void) { return 102; }

clq_status clq_build_permutation(const float* host_scores, int32_t K, int32_t* host_perm) {
  if (host_scores == nullptr || host_perm == nullptr || K < 1) return CLQ_ERR_INVALID_ARG;
  for (int32_t k = 0; k < K; ++k)
    if (std::isnan(host_scores[k])) return CLQ_ERR_INVALID_ARG;
  std::vector<int32_t> order(K);
  std::iota(order.begin(), order.end(), 0);
  std::sort(order.begin(), order.end(), [&](int32_t a, int32_t c) {
    if (host_scores[a] != host_scores[c]) return host_scores[a] > host_scores[c];
    return a < c;
  });
  std::vector<char> high(K, 0);
  for (int32_t i = 0; i < K / 2; ++i) high[order[i]] = 1;
  int32_t pos = 0;
  for (int32_t k = 0; k < K; ++k)
    if (high[k]) host_perm[pos++] = k;
  for (int32_t k = 0; k < K; ++k)
    if (!high[k]) host_perm[pos++] = k;
  return CLQ_OK;
}

clq_status clq_outlier_scores(const void* calib, clq_dtype dtype, int32_t B, int32_t T,
                              int32_t K, float* scores, void* stream) {
  if (!valid_dtype(dtype) || B < 1 || T < 1 || K < 1) return CLQ_ERR_INVALID_ARG;
  if (calib == nullptr || scores == nullptr) return CLQ_ERR_INVALID_ARG;
  if (!aligned(calib, 2) || !aligned(scores, 4)) return CLQ_ERR_ALIGN;
  int32_t* status = nullptr;
  clq_status st = device_setup(&status);
  if (st != CLQ_OK) return st;
  return from_cuda(
      clq::launch_outlier_scores(calib, dtype, B, T, K, scores, static_cast<cudaStream_t>(stream)));
}

clq_status clq_outlier_scores_metric(const void* calib, clq_dtype dtype, int32_t B, int32_t T,
                                     int32_t K, clq_outlier_metric metric, float* scores,
                                     void* stream) {
  if (!valid_dtype(dtype) || B < 1 || T < 1 || K < 1) return CLQ_ERR_INVALID_ARG;
  if (static_cast<int>(metric) < CLQ_METRIC_ABSMAX || static_cast<int>(metric) > CLQ_METRIC_PAR)
    return CLQ_ERR_INVALID_ARG;
  if (T > 16384) return CLQ_ERR_SHAPE;
  if (calib == nullptr || scores == nullptr) return CLQ_ERR_INVALID_ARG;
  if (!aligned(calib, 2) || !aligned(scores, 4)) return CLQ_ERR_ALIGN;
  int32_t* status = nullptr;
  clq_status st = device_setup(&status);
  if (st != CLQ_OK) return st;
  return from_cuda(clq::launch_outlier_metric(calib, dtype, B, T, K, static_cast<int>(metric),
                                              scores, static_cast<cudaStream_t>(stream)));
}

clq_status clq_prepare_weights(const void* W, clq_dtype dtype, int32_t N, int32_t K, int32_t ldw,
                               const int32_t* perm, int32_t b, const float* clip, uint8_t* Wq,
                               float* s_w, float* w_rot_dbg, void* stream) {
  return rotate_quant_common(W, dtype, N, K, ldw, perm, b, clip, CLQ_CODES_INT4_PACKED, Wq, s_w,
                             w_rot_dbg, stream, nullptr, true);
}

clq_status clq_prepare_weights_codes(const void* W, clq_dtype dtype, int32_t N, int32_t K,
                                     int32_t ldw, const int32_t* perm, int32_t b,
                                     const float* clip, clq_codes w_codes, uint8_t* Wq,
                                     float* s_w, float* w_rot_dbg, void* stream) {
  return rotate_quant_common(W, dtype, N, K, ldw, perm, b, clip, w_codes, Wq, s_w, w_rot_dbg,
                             stream, nullptr, true);
}

clq_status clq_rotate_quant_act(const void* X, clq_dtype dtype, int32_t M, int32_t K, int32_t ldx,
                                const int32_t* perm, int32_t b, clq_codes x_codes, uint8_t* Xq,
                                float* s_x, float* x_rot_dbg, void* stream) {
  return rotate_quant_common(X, dtype, M, K, ldx, perm, b, nullptr, x_codes, Xq, s_x, x_rot_dbg,
                             stream);
}

clq_status clq_rotate_quant_act_asym(const void* X, clq_dtype dtype, int32_t M, int32_t K,
                                     int32_t ldx, const int32_t* perm, int32_t b,
                                     clq_codes x_codes, uint8_t* Xq, float* delta, float* lo,
                                     float* x_rot_dbg, void* stream) {
  if (M > 0 && lo == nullptr) return CLQ_ERR_INVALID_ARG;
  return rotate_quant_common(X, dtype, M, K, ldx, perm, b, nullptr, x_codes, Xq, delta,
                             x_rot_dbg, stream, lo);
}

clq_status clq_expand_weights(const uint8_t* Wq, int32_t N, int32_t K, uint8_t* We,
                              void* stream) {
  if (N < 0 || K < 0) return CLQ_ERR_INVALID_ARG;
  if (K < 32 || K > 16384 || K % 32 != 0) return CLQ_ERR_SHAPE;
  if (N == 0) return CLQ_OK;
  if (Wq == nullptr || We == nullptr) return CLQ_ERR_INVALID_ARG;
  if (!aligned(Wq, 16) || !aligned(We, 16)) return CLQ_ERR_ALIGN;
  int32_t* status = nullptr;
  clq_status st = device_setup(&status);
  if (st != CLQ_OK) return st;
  return from_cuda(clq::launch_expand_weights(Wq, N, K, We, static_cast<cudaStream_t>(stream)));
}

clq_status clq_convert_codes(const uint8_t* src, clq_codes src_codes, uint8_t* dst,
                             clq_codes dst_codes, int32_t rows, int32_t K, void* stream) {
  if (!valid_codes(src_codes) || !valid_codes(dst_codes) || rows < 0 || K < 0)
    return CLQ_ERR_INVALID_ARG;
  if (K < 32 || K > 16384 || K % 32 != 0) return CLQ_ERR_SHAPE;
  if ((src_codes == CLQ_CODES_E2M3 || dst_codes == CLQ_CODES_E2M3) && K % 128 != 0)
    return CLQ_ERR_SHAPE;
  if (rows == 0) return CLQ_OK;
  if (src == nullptr || dst == nullptr) return CLQ_ERR_INVALID_ARG;
  if (!aligned(src, 16) || !aligned(dst, 16)) return CLQ_ERR_ALIGN;
  clq_status st = check_e2m3(src_codes, K, src);
  if (st != CLQ_OK || (st = check_e2m3(dst_codes, K, dst)) != CLQ_OK) return st;
  int32_t* status = nullptr;
  st = device_setup(&status);
  if (st != CLQ_OK) return st;
  return from_cuda(clq::launch_convert_codes(src, src_codes, dst, dst_codes, rows, K, status,
                                             static_cast<cudaStream_t>(stream)));
}

clq_status clq_w4a4_linear(const uint8_t* Xq, clq_codes x_codes, const float* s_x,
                           const uint8_t* W, clq_codes w_codes, const float* s_w,
                           const void* bias, int32_t M, int32_t N, int32_t K, int32_t b,
                           clq_dtype out_dtype, void* Y, int32_t* acc_dbg, void* stream) {
  if (!valid_codes(x_codes) || !valid_codes(w_codes)) return CLQ_ERR_INVALID_ARG;
  return clq_linear(Xq, x_codes, s_x, W, w_codes, s_w, bias, M, N, K, b, out_dtype, Y, acc_dbg,
                    stream);
}

clq_status clq_linear(const uint8_t* Xq, clq_codes x_codes, const float* s_x, const uint8_t* W,
                      clq_codes w_codes, const float* s_w, const void* bias, int32_t M,
                      int32_t N, int32_t K, int32_t b, clq_dtype out_dtype, void* Y,
                      int32_t* acc_dbg, void* stream) {
  return linear_common(Xq, x_codes, s_x, nullptr, W, w_codes, s_w, nullptr, bias, M, N, K, b,
                       out_dtype, Y, acc_dbg, stream);
}

clq_status clq_linear_asym(const uint8_t* Xq, clq_codes x_codes, const float* delta,
                           const float* lo, const uint8_t* W, clq_codes w_codes,
                           const float* s_w, const float* wsum, const void* bias, int32_t M,
                           int32_t N, int32_t K, int32_t b, clq_dtype out_dtype, void* Y,
                           int32_t* acc_dbg, void* stream) {
  if (x_codes == CLQ_CODES_INT4_PACKED || w_codes == CLQ_CODES_INT4_PACKED)
    return valid_any_codes(x_codes) && valid_any_codes(w_codes) ? CLQ_ERR_UNSUPPORTED
                                                                : CLQ_ERR_INVALID_ARG;
  if (M > 0 && N > 0 && (lo == nullptr || wsum == nullptr)) return CLQ_ERR_INVALID_ARG;
  return linear_common(Xq, x_codes, delta, lo, W, w_codes, s_w, wsum, bias, M, N, K, b,
                       out_dtype, Y, acc_dbg, stream);
}

clq_status clq_weight_code_sums(const uint8_t* W, clq_codes w_codes, int32_t N, int32_t K,
                                float* wsum, void* stream) {
  if (!valid_any_codes(w_codes) || N < 0) return CLQ_ERR_INVALID_ARG;
  if (K < 32 || K > 16384 || K % 32 != 0) return CLQ_ERR_SHAPE;
  if (w_codes == CLQ_CODES_E2M3 && K % 128 != 0) return CLQ_ERR_SHAPE;
  if (N == 0) return CLQ_OK;
  if (W == nullptr || wsum == nullptr) return CLQ_ERR_INVALID_ARG;
  if (!aligned(W, 16) || !aligned(wsum, 4)) return CLQ_ERR_ALIGN;
  clq_status st = check_e2m3(w_codes, K, W);
  if (st != CLQ_OK) return st;
  int32_t* status = nullptr;
  st = device_setup(&status);
  if (st != CLQ_OK) return st;
  return from_cuda(
      clq::launch_code_sums(W, w_codes, N, K, wsum, static_cast<cudaStream_t>(stream)));
}

}  // extern "C"

namespace clq {

// Host checks of clq_fused_linear's arguments other than its workspace, in
// the order that call makes them; *noop is set when M or N is 0.
int32_t fused_linear_check(const void* X, int32_t dtype, int32_t M, int32_t K, int32_t ldx,
                           const int32_t* perm, int32_t b, const uint8_t* W, int32_t w_codes,
                           const float* s_w, const void* bias, int32_t N, const void* Y,
                           bool* noop) {
  *noop = false;
  if (!valid_dtype(dtype) || !valid_codes(w_codes) || M < 0 || N < 0)
    return CLQ_ERR_INVALID_ARG;
  clq_status st = check_k_b(K, b);
  if (st != CLQ_OK) return st;
  if (w_codes == CLQ_CODES_E2M3 && K % 128 != 0) return CLQ_ERR_SHAPE;
  if (ldx < K) return CLQ_ERR_SHAPE;
  if (ldx % 8 != 0) return CLQ_ERR_ALIGN;
  if (M == 0 || N == 0) {
    *noop = true;
    return CLQ_OK;
  }
  if (X == nullptr || perm == nullptr || W == nullptr || s_w == nullptr || Y == nullptr)
    return CLQ_ERR_INVALID_ARG;
  if (!aligned(X, 16) || !aligned(W, 16) || !aligned(Y, 16) || !aligned(perm, 4) ||
      !aligned(s_w, 4) || (bias != nullptr && !aligned(bias, 2)))
    return CLQ_ERR_ALIGN;
  return check_e2m3(w_codes, K, W);
}

int32_t device_check() {
  int32_t* status = nullptr;
  return device_setup(&status);
}

}  // namespace clq

extern "C" {

size_t clq_fused_linear_workspace_size(int32_t M, int32_t K) {
  if (M < 0 || K < 32 || K > 16384 || K % 32 != 0) return 0;
  return clq::fused_workspace_layout(M, K).bytes;
}

clq_status clq_fused_linear(const void* X, clq_dtype dtype, int32_t M, int32_t K, int32_t ldx,
                            const int32_t* perm, int32_t b, const uint8_t* W,
                            clq_codes w_codes, const float* s_w, const void* bias, int32_t N,
                            void* Y, void* workspace, size_t workspace_bytes, void* stream) {
  bool noop = false;
  clq_status st =
      clq::fused_linear_check(X, dtype, M, K, ldx, perm, b, W, w_codes, s_w, bias, N, Y, &noop);
  if (st != CLQ_OK || noop) return st;
  if (workspace == nullptr) return CLQ_ERR_INVALID_ARG;
  const clq::FusedWorkspace ws = clq::fused_workspace_layout(M, K);
  if (workspace_bytes < ws.bytes) return CLQ_ERR_INVALID_ARG;
  if (!aligned(workspace, 256)) return CLQ_ERR_ALIGN;
  int32_t* status = nullptr;
  st = device_setup(&status);
  if (st != CLQ_OK) return st;
  return fused_common(X, dtype, M, K, ldx, perm, b, W, w_codes, s_w, bias, N, Y,
                      static_cast<uint8_t*>(workspace), ws, status, stream);
}

clq_status clq_get_device_status(void* stream, int32_t* out) {
  if (out == nullptr) return CLQ_ERR_INVALID_ARG;
  int32_t* status = nullptr;
  clq_status st = device_setup(&status);
  if (st != CLQ_OK) return st;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if (cudaStreamSynchronize(s) != cudaSuccess) return CLQ_ERR_CUDA;
  int32_t v = 0;
  if (cudaMemcpyAsync(&v, status, sizeof(v), cudaMemcpyDeviceToHost, s) != cudaSuccess ||
      cudaMemsetAsync(status, 0, sizeof(int32_t), s) != cudaSuccess ||
      cudaStreamSynchronize(s) != cudaSuccess)
    return CLQ_ERR_CUDA;
  *out = v;
  return CLQ_OK;
}

clq_status clq_selftest_bounded_wait(int64_t timeout_ns, void* stream) {
  if (timeout_ns < 1000 || timeout_ns > 1000000000) return CLQ_ERR_INVALID_ARG;
  int32_t* status = nullptr;
  clq_status st = device_setup(&status);
  if (st != CLQ_OK) return st;
  return from_cuda(clq::launch_wait_selftest(static_cast<uint64_t>(timeout_ns), status,
                                             static_cast<cudaStream_t>(stream)));
}

clq_status clq_peak_tcgen05_e4m3(int32_t iters, int64_t* ops, void* stream) {
  if (ops == nullptr || iters < 1 || iters > 1000000) return CLQ_ERR_INVALID_ARG;
  int32_t* status = nullptr;
  clq_status st = device_setup(&status);
  if (st != CLQ_OK) return st;
  long long n = 0;
  st = from_cuda(clq::launch_peak_tcgen05(iters, status, static_cast<cudaStream_t>(stream), &n));
  *ops = n;
  return st;
}

clq_status clq_peak_mma_sync(int32_t kind, int32_t iters, int64_t* ops, void* stream) {
  if (ops == nullptr || kind < 0 || kind > 2 || iters < 1 || iters > 1000000)
    return CLQ_ERR_INVALID_ARG;
  int32_t* status = nullptr;
  clq_status st = device_setup(&status);
  if (st != CLQ_OK) return st;
  long long n = 0;
  st = from_cuda(
      clq::launch_peak_mma_sync(kind, iters, status, static_cast<cudaStream_t>(stream), &n));
  *ops = n;
  return st;
}

clq_status clq_peak_hbm_read(const void* buf, uint64_t bytes, int64_t* ops, void* stream) {
  if (ops == nullptr || buf == nullptr || bytes == 0 || bytes % 16 != 0)
    return CLQ_ERR_INVALID_ARG;
  if (reinterpret_cast<uintptr_t>(buf) % 16 != 0) return CLQ_ERR_ALIGN;
  int32_t* status = nullptr;
  clq_status st = device_setup(&status);
  if (st != CLQ_OK) return st;
  st = from_cuda(clq::launch_peak_hbm_read(buf, bytes, status, static_cast<cudaStream_t>(stream)));
  *ops = static_cast<int64_t>(bytes);
  return st;
}

clq_status clq_peak_rq_stream(const void* X, int32_t M, int32_t K, uint8_t* Q, float* S,
                              int64_t* ops, void* stream) {
  if (ops == nullptr || X == nullptr || Q == nullptr || S == nullptr) return CLQ_ERR_INVALID_ARG;
  if (M < 1 || K < 64 || K > 16384 || K % 64 != 0) return CLQ_ERR_SHAPE;
  if (!aligned(X, 16) || !aligned(Q, 16) || !aligned(S, 4)) return CLQ_ERR_ALIGN;
  int32_t* status = nullptr;
  clq_status st = device_setup(&status);
  if (st != CLQ_OK) return st;
  long long bytes = 0;
  st = from_cuda(clq::launch_peak_rq_stream(X, M, K, Q, S, status,
                                            static_cast<cudaStream_t>(stream), &bytes));
  *ops = bytes;
  return st;
}

clq_status clq_peak_operand_stream(const uint8_t* buf, int32_t rows, int32_t K,
                                   clq_codes codes, int32_t mma, int32_t tiles, int64_t* ops,
                                   void* stream) {
  if (ops == nullptr || buf == nullptr || (codes != CLQ_CODES_E4M3 && codes != CLQ_CODES_E2M3) ||
      mma < 0 || mma > 1 || tiles < 1 || tiles > 100000)
    return CLQ_ERR_INVALID_ARG;
  if (rows < 256 || rows % 256 != 0 || K < 128 || K > 16384 || K % 128 != 0)
    return CLQ_ERR_SHAPE;
  if (reinterpret_cast<uintptr_t>(buf) % 32 != 0) return CLQ_ERR_ALIGN;
  int32_t* status = nullptr;
  clq_status st = device_setup(&status);
  if (st != CLQ_OK) return st;
  long long bytes = 0, macs = 0;
  st = from_cuda(clq::launch_peak_operand_stream(buf, rows, K, codes, mma, tiles, status,
                                                 static_cast<cudaStream_t>(stream), &bytes,
                                                 &macs));
  *ops = mma == 1 ? macs : bytes;
  return st;
}

size_t clq_clip_search_workspace_size(int32_t M, int32_t N, int32_t K, const float* host_grid,
                                      int32_t G) {
  if (M < 1 || N < 1 || K < 32 || K > 16384 || K % 32 != 0 || G < 1 || host_grid == nullptr)
    return 0;
  for (int g = 0; g < G; ++g)
    if (!(host_grid[g] >= 0.f && host_grid[g] < 1.f)) return 0;
  return clip_workspace_layout(M, N, K, clip_table_width(K, host_grid, G), G).bytes;
}

clq_status clq_clip_search(const void* W, clq_dtype dtype, int32_t N, int32_t K, int32_t ldw,
                           const int32_t* perm, int32_t b, const void* Xcal, int32_t M,
                           int32_t ldx, const float* Yref, const void* bias,
                           const float* host_grid, int32_t G, float* clip_out,
                           double* host_errors, int32_t* host_best, void* workspace,
                           size_t workspace_bytes, void* stream) {
  if (!valid_dtype(dtype) || N < 1 || M < 1 || G < 1) return CLQ_ERR_INVALID_ARG;
  clq_status st = check_k_b(K, b);
  if (st != CLQ_OK) return st;
  if (ldw < K || ldx < K) return CLQ_ERR_SHAPE;
  if (ldw % 8 != 0 || ldx % 8 != 0) return CLQ_ERR_ALIGN;
  if (W == nullptr || perm == nullptr || Xcal == nullptr || Yref == nullptr ||
      host_grid == nullptr || clip_out == nullptr || host_errors == nullptr ||
      host_best == nullptr || workspace == nullptr)
    return CLQ_ERR_INVALID_ARG;
  for (int g = 0; g < G; ++g)
    if (!(host_grid[g] >= 0.f && host_grid[g] < 1.f)) return CLQ_ERR_INVALID_ARG;
  const int J = clip_table_width(K, host_grid, G);
  const ClipWorkspace ws = clip_workspace_layout(M, N, K, J, G);
  if (workspace_bytes < ws.bytes) return CLQ_ERR_INVALID_ARG;
  if (!aligned(W, 16) || !aligned(Xcal, 16) || !aligned(perm, 4) || !aligned(Yref, 4) ||
      !aligned(clip_out, 4) || (bias != nullptr && !aligned(bias, 2)) ||
      !aligned(workspace, 256))
    return CLQ_ERR_ALIGN;
  int32_t* status = nullptr;
  st = device_setup(&status);
  if (st != CLQ_OK) return st;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  uint8_t* base = static_cast<uint8_t*>(workspace);
  float* w_rot = reinterpret_cast<float*>(base + ws.w_rot);
  uint8_t* wq = base + ws.wq;
  float* s_w = reinterpret_cast<float*>(base + ws.s_w);
  float* table = reinterpret_cast<float*>(base + ws.table);
  float* clip = reinterpret_cast<float*>(base + ws.clip);
  uint8_t* xq = base + ws.xq;
  float* s_x = reinterpret_cast<float*>(base + ws.s_x);
  void* yh = base + ws.yh;
  double* partial = reinterpret_cast<double*>(base + ws.partial);
  double* errors = reinterpret_cast<double*>(base + ws.errors);

  auto rq = [&](const void* X, int rows, int ld, const float* c, uint8_t* Q, float* S,
                float* rot) {
    clq::RotateQuantArgs a{};
    a.X = X;
    a.M = rows;
    a.K = K;
    a.ld = ld;
    a.perm = perm;
    a.clip = c;
    a.Q = Q;
    a.S = S;
    a.rot = rot;
    a.status = status;
    a.serial = X == W ? 1 : 0;  // the weights: see clq_prepare_weights
    a.logb = log2i(b);
    a.e4m3 = 1;
    return clq::launch_rotate_quant(a, dtype, log2i(b), s);
  };
  // W~ (unclipped) and its table of largest magnitudes; the calibration
  // activations' codes, which every grid point reuses.
  cudaError_t e = rq(W, N, ldw, nullptr, wq, s_w, w_rot);
  if (e == cudaSuccess) e = clq::launch_clip_table(w_rot, N, K, J, table, s);
  if (e == cudaSuccess) e = rq(Xcal, M, ldx, nullptr, xq, s_x, nullptr);
  clq::GemmArgs g{};
  g.s_x = s_x;
  g.s_w = s_w;
  g.bias = bias;
  g.Y = yh;
  g.M = M;
  g.N = N;
  g.K = K;
  g.inv_b = 1.0f / static_cast<float>(b);
  g.status = status;
  for (int gi = 0; gi < G && e == cudaSuccess; ++gi) {
    const int j = static_cast<int>(std::floor(static_cast<double>(host_grid[gi]) * K));
    e = clq::launch_clip_gather(table, N, J, j, clip, s);
    if (e == cudaSuccess) e = rq(W, N, ldw, clip, wq, s_w, nullptr);
    if (e == cudaSuccess)
      e = clq::launch_w4a4_gemm(xq, CLQ_CODES_E4M3, wq, CLQ_CODES_E4M3, g, dtype, s);
    if (e == cudaSuccess)
      e = clq::launch_sq_err_partial(yh, dtype, Yref, static_cast<size_t>(M) * N,
                                     partial + static_cast<size_t>(gi) * kClipPartials,
                                     kClipPartials, s);
  }
  if (e == cudaSuccess) e = clq::launch_sum_partials(partial, G, kClipPartials, errors, s);
  if (e == cudaSuccess)
    e = cudaMemcpyAsync(host_errors, errors, static_cast<size_t>(G) * sizeof(double),
                        cudaMemcpyDeviceToHost, s);
  if (e == cudaSuccess) e = cudaStreamSynchronize(s);
  if (e != cudaSuccess) {
    // Nothing launched before the failure may still use the workspace when
    // the caller regains control.
    cudaStreamSynchronize(s);
    return CLQ_ERR_CUDA;
  }
  int best = 0;
  for (int gi = 1; gi < G; ++gi)
    if (host_errors[gi] < host_errors[best]) best = gi;  // ties: the smaller p
  *host_best = best;
  const int jb = static_cast<int>(std::floor(static_cast<double>(host_grid[best]) * K));
  return from_cuda(clq::launch_clip_gather(table, N, J, jb, clip_out, s));
}

}  // extern "C"
