// Host-side launch interface between the C ABI (clq_api.cu) and the kernels.
#pragma once

#include <algorithm>
#include <cstddef>
#include <cstdint>
#include <utility>
#include <cuda.h>
#include <cuda_runtime.h>

namespace clq {

struct RotateQuantArgs {
  const void* X;         // [M][ld] fp16 / bf16
  int32_t M, K, ld;
  const int32_t* perm;   // [K]
  const float* clip;     // [M] or null (weights only)
  uint8_t* Q;            // [M][K/2] packed, [M][K] E4M3, or [M][2][K] split planes
  float* S;              // [M] scales (asymmetric: delta)
  float* lo;             // [M] row minima (asymmetric codes), or null (symmetric)
  float* rot;            // [M][K] or null
  int32_t rows_per_tile; // filled in by the launcher
  int32_t* status;       // device status word
  int32_t logb;          // log2(b)
  int32_t e4m3;          // codes layout: 0 packed nibbles, 1 one E4M3 byte each,
                         // 2 8-bit codes as two E4M3 planes (16 h, l), 3 E2M3
                         // (16 codes in 12 bytes)
  int32_t serial;        // 1: launched without programmatic overlap (weight
                         // preparation, whose swap vector may have just been
                         // written on the device)
};

cudaError_t launch_rotate_quant(const RotateQuantArgs& a, int dtype, int logb,
                                cudaStream_t st);
void rotate_quant_config(int M, int K, int sms, int* rows_per_tile, int* threads,
                         size_t* smem);
cudaError_t launch_outlier_scores(const void* calib, int dtype, int B, int T, int K,
                                  float* scores, cudaStream_t st);
cudaError_t launch_outlier_metric(const void* calib, int dtype, int B, int T, int K, int metric,
                                  float* scores, cudaStream_t st);

struct GemmArgs {
  const float* s_x;   // [M]
  const float* s_w;   // [N]
  const void* bias;   // [N] out dtype, or null
  void* Y;            // [M][N] out dtype
  int32_t* acc_dbg;   // [M][N] or null
  int32_t M, N, K;
  float inv_b;
  int32_t* status;
  // Asymmetric activation codes (centered, q - 2^(n-1)): s_x holds each row's
  // step delta, lo its minimum, wsum[N] the weight-code row sums, zp_shift
  // 2^(n-1).  lo == null: symmetric codes.
  const float* lo;
  const float* wsum;
  float zp_shift;
};

// A = activation codes, B = weight codes, each in layout CLQ_CODES_INT4_PACKED
// ([rows][K/2]), CLQ_CODES_E4M3 ([rows][K]) or, for 8-bit codes,
// CLQ_CODES_E4M3_SPLIT ([rows][2][K]; A split with B E4M3 or split); TMA maps
// are built here.
// Output-channel tile width (192 or 256) of the E4M3 x E4M3 GEMM for an
// M x N product on `sms` SMs.
int gemm_tile_n(int M, int N, int sms);
cudaError_t launch_w4a4_gemm(const uint8_t* Xq, int x_codes, const uint8_t* W, int w_codes,
                             const GemmArgs& g, int out_dtype, cudaStream_t st);

// Clip search (clip_search.cu): table[n][j] = j-th largest |w_rot[n][:]|
// (j < J); clip[n] = table[n][j]; partial[b] = block b's share of
// sum (yh - yref)^2 in fp64 over n elements (P blocks); out[g] = the fixed-order
// sum of partial[g][0 .. P).
cudaError_t launch_clip_table(const float* w_rot, int N, int K, int J, float* table,
                              cudaStream_t st);
cudaError_t launch_clip_gather(const float* table, int N, int J, int j, float* clip,
                               cudaStream_t st);
cudaError_t launch_sq_err_partial(const void* yh, int dtype, const float* yref, size_t n,
                                  double* partial, int P, cudaStream_t st);
cudaError_t launch_sum_partials(const double* partial, int G, int P, double* out,
                                cudaStream_t st);

// wsum[n] = sum_k of the integer codes of row n, any layout (exact in fp32).
cudaError_t launch_code_sums(const uint8_t* W, int codes, int N, int K, float* wsum,
                             cudaStream_t st);

cudaError_t launch_expand_weights(const uint8_t* Wq, int N, int K, uint8_t* We, cudaStream_t st);
// rows x K codes from one 4-bit layout to another (K % 16 == 0; E2M3 needs
// K % 128 == 0 only for the GEMM's tensor maps).
cudaError_t launch_convert_codes(const uint8_t* src, int src_codes, uint8_t* dst, int dst_codes,
                                 int rows, int K, int32_t* status, cudaStream_t st);

// Workspace of the fused kernel: codes, scales, per-token-block row counters.
struct FusedWorkspace {
  size_t codes_off, scales_off, ready_off, bytes;
};
FusedWorkspace fused_workspace_layout(int M, int K);

// Fused rotate-quant + GEMM: `rq` describes the activation side (its Q / S
// point into the workspace), `g` the product (s_x = workspace scales).
cudaError_t launch_fused_linear(const RotateQuantArgs& rq, const uint8_t* W, int w_codes,
                                const GemmArgs& g, int logb, int dtype, uint32_t* ready,
                                cudaStream_t st);

// Host checks of clq_fused_linear's arguments other than its workspace, in
// the order that call makes them (a clq_status; *noop set when M or N is 0),
// and the check that the current device is an sm_103 GPU.
int32_t fused_linear_check(const void* X, int32_t dtype, int32_t M, int32_t K, int32_t ldx,
                           const int32_t* perm, int32_t b, const uint8_t* W, int32_t w_codes,
                           const float* s_w, const void* bias, int32_t N, const void* Y,
                           bool* noop);
int32_t device_check();

// Bounded-wait self test (one CTA, one mbarrier nothing arrives at).
cudaError_t launch_wait_selftest(uint64_t timeout_ns, int32_t* status, cudaStream_t st);

// cuTensorMapEncodeTiled through the runtime's driver entry point.
bool encode_tma_2d(CUtensorMap* map, CUtensorMapDataType dt, uint32_t esize, const void* base,
                   uint64_t inner, uint64_t rows, uint32_t box_inner, uint32_t box_rows,
                   CUtensorMapSwizzle swz);
bool encode_tma_2d_strided(CUtensorMap* map, CUtensorMapDataType dt, uint32_t esize,
                           const void* base, uint64_t inner, uint64_t rows,
                           uint64_t row_stride_bytes, uint32_t box_inner, uint32_t box_rows,
                           CUtensorMapSwizzle swz);
bool encode_tma_2d_u8(CUtensorMap* map, const void* base, uint64_t inner_bytes,
                      uint64_t rows, uint32_t box_inner, uint32_t box_rows);
// 2-byte output tile map for the epilogue stores (box 32 columns x 128 rows).
bool encode_tma_out_tile(CUtensorMap* map, void* Y, int M, int N);
int sm_count();  // cached per device
// TMA map of a code array (rows x K) in layout `codes`, box_rows rows; for
// the split layout, of plane `plane` (0 or 1).
bool encode_codes_map(CUtensorMap* map, const uint8_t* base, int codes, int rows, int K,
                      int box_rows, int plane);
// Peak-rate microbenchmarks (peaks.cu); *macs / *ops receive the work done.
cudaError_t launch_peak_tcgen05(int iters, int32_t* status, cudaStream_t st, long long* macs);
cudaError_t launch_peak_mma_sync(int kind, int iters, int32_t* sink, cudaStream_t st,
                                 long long* macs);
cudaError_t launch_peak_hbm_read(const void* buf, size_t bytes, int32_t* sink, cudaStream_t st);
// The GEMM's operand stream (peaks.cu): `tiles` 128 x 256 tiles a CTA, one
// CTA per SM, from a rows x K code array (E4M3 or E2M3); with `mma` the MMAs
// too.  *smem_bytes / *macs receive the shared-memory bytes filled and the
// multiply-accumulates.
cudaError_t launch_peak_operand_stream(const uint8_t* buf, int rows, int K, int codes, int mma,
                                       int tiles, int32_t* status, cudaStream_t st,
                                       long long* smem_bytes, long long* macs);
// Raise `func`'s dynamic shared-memory limit to the device maximum once per
// device, and (per_sm != null) return its occupancy for (threads, smem),
// cached, so that launches make no per-call attribute queries.
cudaError_t kernel_setup(const void* func, size_t smem, int threads, int* per_sm);

// Launch with programmatic stream serialization (pdl true): the kernel may
// start while the previous kernel on `st` finishes and must call pdl_wait()
// before it reads what that kernel may have written.  (Only kernel-to-kernel
// edges overlap; after a copy or a memset the launch waits as usual.)  With
// pdl false the launch waits for the previous kernel as usual.
template <typename... KArgs, typename... Args>
cudaError_t launch_ex(void (*kernel)(KArgs...), int grid, int threads, size_t smem,
                      cudaStream_t st, bool pdl, Args&&... args) {
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(static_cast<unsigned>(grid));
  cfg.blockDim = dim3(static_cast<unsigned>(threads));
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, kernel, std::forward<Args>(args)...);
}

template <typename... KArgs, typename... Args>
cudaError_t launch_pdl(void (*kernel)(KArgs...), int grid, int threads, size_t smem,
                       cudaStream_t st, Args&&... args) {
  return launch_ex(kernel, grid, threads, smem, st, true, std::forward<Args>(args)...);
}

}  // namespace clq
