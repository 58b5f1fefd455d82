/*
 * clq.h - C ABI of libclq, the GB300 (sm_103a) inference path of CLQ's
 * W4A4 orthogonal-based-smoothing (OBS) linear layer, arxiv 2509.24416, with
 * the paper's other bit settings (W4A8, W8A8), asymmetric activation codes
 * (Eq. 1), the alternative outlier metrics (Sec. 4.4) and the per-layer clip
 * search (Eq. 3).
 *
 * The layer computes Y = X W^T + bias with both operands quantized to 4 bits
 * (or 8, see clq_linear) after the OBS transform G = S H (Sec. 3.3): S is a
 * column swap stored as an index vector `perm` (position k holds the
 * original column perm[k]) and
 * H = diag(H_b, ..., H_b) with H_b the Sylvester Hadamard matrix of order b,
 * H_b[i][j] = (-1)^popcount(i & j).  G is absorbed into W offline; the
 * activations are rotated online with a fast Walsh-Hadamard transform and
 * quantized per token with dynamic bounds (Sec. 3.1).  Quantization is the
 * symmetric reading of Eq. 1: r = max|row| (optionally clipped), s = r / 7
 * in fp32, q = clamp(rint(v / s), -7, 7), ties to even, code -8 unused
 * (qmax 127 for 8-bit codes; Eq. 1 itself, with dynamic min and max, for
 * clq_rotate_quant_act_asym).
 * H is unnormalized (H_b H_b^T = b I), so the epilogue divides by b once:
 *     Y[i][n] = acc[i][n] * s_x[i] * s_w[n] / b + bias[n],
 *     acc[i][n] = sum_k qx[i][k] * qw[n][k]  (exact integer).
 *
 * Conventions for every call:
 *  - Returns a clq_status; 0 (CLQ_OK) on success.  No exception or abort
 *    crosses the ABI.  Arguments are validated on the host before anything is
 *    launched; on an error nothing is launched and no output is touched.
 *  - Tensor pointers are DEVICE pointers owned by the caller unless the name
 *    starts with host_.  The library allocates, frees and synchronizes
 *    nothing in these calls (clq_get_device_status and the offline
 *    clq_clip_search synchronize by design).
 *  - Launches are asynchronous on `stream` (a cudaStream_t passed as void*;
 *    NULL is the legacy default stream).
 *  - Row-major layouts; `ld*` arguments are row strides in ELEMENTS.
 *  - Packed INT4 rows: byte j holds code 2j in its low nibble and code 2j+1
 *    in its high nibble, 4-bit two's complement.  A packed row of K codes is
 *    K/2 bytes and rows are contiguous (stride K/2).
 *  - Shape rules: 1 <= b <= 256 and b a power of two; K % 32 == 0,
 *    K % b == 0, 32 <= K <= 16384; M, N >= 0 (0 is an empty no-op);
 *    ld* >= K and ld* % 8 == 0.  Matrices and code arrays are 16-byte
 *    aligned; vectors (perm, scales, clip) 4-byte and bias 2-byte aligned.
 *  - Device-side faults the host cannot see (an index in `perm` outside
 *    [0, K), a pipeline wait that exceeds its time limit) are recorded in a
 *    device status word read by clq_get_device_status; the kernel skips the
 *    offending access instead of faulting.
 *  - Stream order holds as usual: every kernel reads its inputs and writes
 *    its outputs only after the work enqueued before it on `stream` has
 *    completed, with one exception below.  The kernels launch with
 *    programmatic dependent launch, so a kernel of this library may become
 *    resident while the previous one on the stream drains; in that window
 *    it sets up on-chip state, hints L2 prefetches of its first input rows
 *    (which change no value it later reads) and, in the activation
 *    rotate-quant calls (clq_rotate_quant_act, clq_rotate_quant_act_asym),
 *    reads the swap vector `perm`, a layer constant.  So that `perm` must not
 *    be written by the kernel enqueued just before the call on the same
 *    stream: the writes of a kernel are guaranteed visible to the next one
 *    only once the latter has waited for it.  No call of this library writes
 *    a swap vector (clq_build_permutation runs on the host); a copy or
 *    another call of this library enqueued between the writing kernel and
 *    the call restores the usual order.  The weight-preparation calls and
 *    clq_clip_search launch without the overlap, so a swap vector computed
 *    on the device just before them is safe.
 *  - The library keeps no per-call state and is safe to call from several
 *    host threads.
 *  - The hot-path calls (rotate-quant, the products, the fused kernel) launch
 *    kernels only, so they can be captured in a CUDA graph; the first call of
 *    each kernel configuration on a device sets the kernel's shared-memory
 *    limit, so make one call of the same shape before capturing.
 */
#ifndef CLQ_H
#define CLQ_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef int32_t clq_status;
#define CLQ_OK 0
#define CLQ_ERR_INVALID_ARG 1 /* null pointer, bad enum, negative size    */
#define CLQ_ERR_SHAPE 2       /* shape rule above violated                 */
#define CLQ_ERR_ALIGN 3       /* pointer or stride not 16-byte aligned     */
#define CLQ_ERR_UNSUPPORTED 4 /* no usable sm_103a device / feature        */
#define CLQ_ERR_CUDA 5        /* a CUDA runtime call failed                */
#define CLQ_ERR_TIMEOUT 6     /* a bounded device-side wait ran out        */
#define CLQ_ERR_DEVICE_INDEX 7 /* perm held an index outside [0, K)        */
#define CLQ_ERR_SCRATCH_LIMIT 8 /* problem needs more than the static     */
                                /* scratch of clq_fused_linear_noalloc     */
#define CLQ_ERR_DEVICE_CODE 9  /* a code array held a value outside the   */
                               /* INT4 range [-7, 7] (clq_convert_codes)   */

typedef int32_t clq_dtype;
#define CLQ_F16 0
#define CLQ_BF16 1

/*
 * Layout of an array of codes (activations or weights), `rows` x K.  The
 * 4-bit layouts:
 *  CLQ_CODES_INT4_PACKED  [rows][K/2] bytes, two codes per byte (code 2j in
 *                         the low nibble), 4-bit two's complement; the
 *                         storage format.
 *  CLQ_CODES_E4M3         [rows][K] bytes, one code per byte holding the
 *                         code's exact E4M3 encoding (every integer in
 *                         [-7, 7] is an E4M3 value); the execution layout the
 *                         tensor-core GEMM loads with TMA directly, without
 *                         expanding nibbles in every CTA.  A zero code may
 *                         be written as either E4M3 zero (0x00 or 0x80).
 *  CLQ_CODES_E2M3         [rows][3K/4] bytes: each group of 16 consecutive
 *                         codes is one little-endian 96-bit field (12
 *                         bytes), code i of the group in bits 6i .. 6i + 5
 *                         holding the code's exact E2M3 encoding (sign bit
 *                         5, two exponent bits with bias 1, three mantissa
 *                         bits: 0..7 are 0x00, 0x08, 0x10, 0x14, 0x18, 0x1A,
 *                         0x1C, 0x1E; every integer in [-7, 7] is an E2M3
 *                         value).  The tensor-core GEMM's tensor maps pad
 *                         each 12-byte group to 16 bytes on the way into
 *                         shared memory, the layout 6-bit MMA operands take,
 *                         so this execution layout needs 3/4 of E4M3's
 *                         bytes.  Requires K % 128 == 0 and 32-byte aligned
 *                         arrays.  A zero code may be written as either E2M3
 *                         zero (0x00 or 0x20).  The GEMM takes it for both
 *                         operands together.
 * The codes are the same INT4 values in every layout and every call gives
 * identical results for any of them.  The 8-bit layout (the W4A8 and W8A8 bit
 * settings of Sec. 4.1; codes q in [-127, 127], s = r / 127):
 *  CLQ_CODES_E4M3_SPLIT   [rows][2][K] bytes: for each row, plane 0 holds the
 *                         E4M3 encoding of 16 h and plane 1 that of l, where
 *                         h = floor((q + 8) / 16) in [-8, 8] and
 *                         l = q - 16 h in [-8, 7]; both are E4M3 values, so
 *                         the tensor cores take q = 16 h + l as two MMAs
 *                         into one accumulator.
 */
typedef int32_t clq_codes;
#define CLQ_CODES_INT4_PACKED 0
#define CLQ_CODES_E4M3 1
#define CLQ_CODES_E4M3_SPLIT 2
#define CLQ_CODES_E2M3 3

/* Human-readable name of a status code (static string, never NULL). */
const char* clq_status_string(clq_status status);

/* ABI version, major * 100 + minor. */
int32_t clq_version(void);

/*
 * Outlier score per input channel (Sec. 3.3, "Data Preparing" and "Outlier
 * Detection"): S = mean over the batch of calib[B][T][K] (fp32, summed over
 * the batch in order, then divided by B), score[k] = max_t |S[t][k]|.
 * calib: device, dtype `dtype`, contiguous [B][T][K].  scores: device fp32
 * [K].  Requires B, T, K >= 1.  Offline; not on the timed path.
 */
clq_status clq_outlier_scores(const void* calib, clq_dtype dtype, int32_t B,
                              int32_t T, int32_t K, float* scores,
                              void* stream);

/*
 * Outlier metrics of Sec. 4.4 ("Choice of Outlier Metric"), which names them
 * and their parameters but no formulas; this library reads them as below,
 * every step in fp32 in a fixed order (the scores decide an integer
 * permutation):
 *   CLQ_METRIC_ABSMAX      max_t |S| (Sec. 3.3, as clq_outlier_scores);
 *   CLQ_METRIC_PERCENTILE  max(|P(1 %)|, |P(99 %)|) of S, P by linear
 *                          interpolation between order statistics:
 *                          pos = q (T - 1), v[lo] + (pos - lo)(v[lo + 1] - v[lo]);
 *   CLQ_METRIC_TOPK_MEAN   mean of the k largest |S|, k = max(1, (T + 50) / 100)
 *                          (1 % of the tokens), summed from the largest down;
 *   CLQ_METRIC_RANGE       max_t S - min_t S;
 *   CLQ_METRIC_PAR         peak-to-average ratio max_t |S| / (sum_t |S| / T),
 *                          the sum over t in order; 0 for an all-zero channel.
 */
typedef enum clq_outlier_metric {
  CLQ_METRIC_ABSMAX = 0,
  CLQ_METRIC_PERCENTILE = 1,
  CLQ_METRIC_TOPK_MEAN = 2,
  CLQ_METRIC_RANGE = 3,
  CLQ_METRIC_PAR = 4
} clq_outlier_metric;

/*
 * Outlier score per input channel under `metric` (see above), from the batch
 * mean S of calib[B][T][K] (device, dtype `dtype`, contiguous) into scores
 * (device fp32 [K]).  Requires B, K >= 1 and 1 <= T <= 16384
 * (CLQ_ERR_SHAPE beyond).  Offline; not on the timed path.
 */
clq_status clq_outlier_scores_metric(const void* calib, clq_dtype dtype, int32_t B, int32_t T,
                                     int32_t K, clq_outlier_metric metric, float* scores,
                                     void* stream);

/*
 * Column-swap vector from outlier scores (Sec. 3.3, "Outlier Detection"):
 * rank channels by score descending (ties to the lower index); the first
 * K/2 (rounded down) form the high-peak set, placed left, the rest right,
 * each side in ascending channel index.  HOST pointers: host_scores [K],
 * host_perm [K] (written).  Requires K >= 1; NaN scores are rejected.
 */
clq_status clq_build_permutation(const float* host_scores, int32_t K,
                                 int32_t* host_perm);

/*
 * Offline weight preparation (Sec. 3.3, "Overhead Analysis": W~ = G^T-side
 * absorption, here W~ = W_p H with W_p[n][k] = W[n][perm[k]]), then
 * per-output-channel symmetric INT4: s_w[n] = min(max_k |W~[n][k]|,
 * clip[n]) / 7, Wq[n] = pack(clamp(rint(W~[n] / s_w[n]), -7, 7)).
 * W: device [N][ldw] of `dtype`.  perm: device int32 [K].  clip: device fp32
 * [N] (> 0) or NULL for no clipping.  Wq: device uint8 [N][K/2].  s_w:
 * device fp32 [N].  w_rot_dbg: device fp32 [N][K] or NULL; when given it
 * receives W~ (the fp32 rotated rows) for parity checks.
 */
clq_status clq_prepare_weights(const void* W, clq_dtype dtype, int32_t N,
                               int32_t K, int32_t ldw, const int32_t* perm,
                               int32_t b, const float* clip, uint8_t* Wq,
                               float* s_w, float* w_rot_dbg, void* stream);

/*
 * clq_prepare_weights in any code layout (`w_codes`): 4-bit codes (qmax 7)
 * for CLQ_CODES_INT4_PACKED ([N][K/2]), CLQ_CODES_E4M3 ([N][K]) or
 * CLQ_CODES_E2M3 ([N][3K/4], K % 128 == 0, Wq 32-byte aligned), 8-bit
 * codes (qmax 127, the W8A8 setting) for CLQ_CODES_E4M3_SPLIT ([N][2][K]).
 * The clip bound caps max_k |W~[n][k]| as above.
 */
clq_status clq_prepare_weights_codes(const void* W, clq_dtype dtype, int32_t N,
                                     int32_t K, int32_t ldw,
                                     const int32_t* perm, int32_t b,
                                     const float* clip, clq_codes w_codes,
                                     uint8_t* Wq, float* s_w, float* w_rot_dbg,
                                     void* stream);

/*
 * Online activation rotate + quantize (Sec. 3.1 dynamic quantization with
 * Sec. 3.3's online fast Hadamard): X~ = X_p H in fp32, s_x[i] =
 * max_k |X~[i][k]| / qmax, codes clamp(rint(X~[i] / s_x[i]), -qmax, qmax),
 * qmax = 7 for the 4-bit layouts and 127 for CLQ_CODES_E4M3_SPLIT.
 * One HBM pass over X.  X: device [M][ldx] of `dtype`.  perm: device int32
 * [K].  Xq: device uint8 codes in layout `x_codes` ([M][K/2] packed,
 * [M][K] E4M3, [M][3K/4] E2M3 with K % 128 == 0 and Xq 32-byte aligned, or
 * [M][2][K] split).  s_x: device fp32 [M].  x_rot_dbg:
 * device fp32 [M][K] or NULL (receives X~).
 */
clq_status clq_rotate_quant_act(const void* X, clq_dtype dtype, int32_t M,
                                int32_t K, int32_t ldx, const int32_t* perm,
                                int32_t b, clq_codes x_codes, uint8_t* Xq,
                                float* s_x, float* x_rot_dbg, void* stream);

/*
 * Packed INT4 codes [N][K/2] (CLQ_CODES_INT4_PACKED) -> the E4M3 execution
 * layout [N][K] (CLQ_CODES_E4M3).  The codes are unchanged; only the
 * container widens to 8 bits.  Used offline, once per layer, on the weights
 * (weights are static, so expanding them in every CTA of every call would
 * only repeat work).  Wq: device [N][K/2]; We: device [N][K].  Requires
 * N >= 0, K % 32 == 0, K <= 16384.
 */
clq_status clq_expand_weights(const uint8_t* Wq, int32_t N, int32_t K,
                              uint8_t* We, void* stream);

/*
 * A code array of `rows` x K INT4 codes from one 4-bit layout to another
 * (CLQ_CODES_INT4_PACKED, CLQ_CODES_E4M3, CLQ_CODES_E2M3, in any direction,
 * the same layout included).  The codes are unchanged; this is how the
 * storage format (packed nibbles) and the execution layouts are turned into
 * one another, offline.  src: device, [rows][width(src_codes)] bytes; dst:
 * device, [rows][width(dst_codes)] bytes, not overlapping src; width is K/2,
 * K or 3K/4.  Requires rows >= 0, K % 32 == 0, K <= 16384 (K % 128 == 0 when
 * either side is E2M3); arrays 16-byte aligned (32 for E2M3).  A source code
 * outside [-7, 7] (packed -8, or an E4M3 / E2M3 field that holds no integer
 * in that range) is written as 0 and reported as CLQ_ERR_DEVICE_CODE in the
 * device status word.
 */
clq_status clq_convert_codes(const uint8_t* src, clq_codes src_codes,
                             uint8_t* dst, clq_codes dst_codes, int32_t rows,
                             int32_t K, void* stream);

/*
 * INT4 x INT4 product with the dequant + bias epilogue:
 * Y[i][n] = out_dtype(acc[i][n] * s_x[i] * s_w[n] / b + bias[n]).
 * Xq: device activation codes in layout `x_codes` ([M][K/2], [M][K] or
 * [M][3K/4]); s_x: device fp32 [M]; W: device weight codes in layout
 * `w_codes` ([N][K/2], [N][K] or [N][3K/4]); s_w: device fp32 [N]; bias:
 * device [N] of `out_dtype` or NULL; Y: device [M][N] of `out_dtype`.
 * acc_dbg: device int32 [M][N] or NULL; when given it receives the exact
 * integer accumulators.  Packed and E4M3 operands combine in all four ways;
 * CLQ_CODES_E2M3 goes with CLQ_CODES_E2M3 only (other pairings with it return
 * CLQ_ERR_UNSUPPORTED).  Every combination gives identical results.
 */
clq_status clq_w4a4_linear(const uint8_t* Xq, clq_codes x_codes,
                           const float* s_x, const uint8_t* W,
                           clq_codes w_codes, const float* s_w,
                           const void* bias, int32_t M, int32_t N, int32_t K,
                           int32_t b, clq_dtype out_dtype, void* Y,
                           int32_t* acc_dbg, void* stream);

/*
 * The product at any of the paper's bit settings (Sec. 4.1), with the same
 * epilogue as clq_w4a4_linear: Y[i][n] = out_dtype(acc[i][n] * s_x[i] *
 * s_w[n] / b + bias[n]), acc[i][n] = sum_k qx[i][k] * qw[n][k].
 *  W4A4  x_codes and w_codes 4-bit layouts (as clq_w4a4_linear);
 *  W4A8  x_codes CLQ_CODES_E4M3_SPLIT, w_codes CLQ_CODES_E4M3;
 *  W8A8  both CLQ_CODES_E4M3_SPLIT.
 * Other combinations return CLQ_ERR_UNSUPPORTED.  The accumulators are
 * exact integers for every K <= 16384 at every setting (W8A8 keeps its plane
 * products in three accumulators and adds them as integers).  acc_dbg (int32
 * [M][N] or NULL) receives them.  Arguments otherwise as for
 * clq_w4a4_linear.
 */
clq_status clq_linear(const uint8_t* Xq, clq_codes x_codes, const float* s_x,
                      const uint8_t* W, clq_codes w_codes, const float* s_w,
                      const void* bias, int32_t M, int32_t N, int32_t K,
                      int32_t b, clq_dtype out_dtype, void* Y,
                      int32_t* acc_dbg, void* stream);

/*
 * Asymmetric activation quantization (Eq. 1 with dynamic bounds, Sec. 3.1):
 * after the same rotation as clq_rotate_quant_act, each token row X~[i] is
 * quantized with l = min_k X~[i][k], r = max_k X~[i][k]:
 *   delta[i] = (r - l) / (2^n - 1),
 *   q = rint((X~ - l) / (r - l) * (2^n - 1)) in [0, 2^n - 1], ties to even,
 * and x^ = delta q + l (Eq. 1 as printed omits the + l; this is the reading
 * under which x^ approximates x).  A constant row gets delta = 0, q = 0.
 * The codes are stored CENTERED, c = q - 2^(n-1), so they share the signed
 * containers of the symmetric path: n = 4 for CLQ_CODES_INT4_PACKED and
 * CLQ_CODES_E4M3 (c in [-8, 7]), n = 8 for CLQ_CODES_E4M3_SPLIT
 * (c in [-128, 127]).  delta, lo: device fp32 [M] (lo receives l).  Other
 * arguments as for clq_rotate_quant_act.
 */
clq_status clq_rotate_quant_act_asym(const void* X, clq_dtype dtype, int32_t M,
                                     int32_t K, int32_t ldx,
                                     const int32_t* perm, int32_t b,
                                     clq_codes x_codes, uint8_t* Xq,
                                     float* delta, float* lo, float* x_rot_dbg,
                                     void* stream);

/*
 * wsum[n] = sum_k qw[n][k], the integer code sums of each weight row, for
 * the zero-point epilogue of clq_linear_asym (exact in fp32: |wsum| <=
 * 127 * 16384).  W: device codes [N][...] in layout `w_codes`; wsum: device
 * fp32 [N].  Offline, once per layer.
 */
clq_status clq_weight_code_sums(const uint8_t* W, clq_codes w_codes, int32_t N,
                                int32_t K, float* wsum, void* stream);

/*
 * The product of asymmetric activations (centered codes from
 * clq_rotate_quant_act_asym, delta, lo) and symmetric weights, with the
 * zero-point epilogue that equals X^ W^^T / b + bias:
 *   Y[i][n] = out_dtype(s_w[n] / b * (delta[i] acc[i][n] + m[i] wsum[n])
 *                       + bias[n]),
 *   acc[i][n] = sum_k c[i][k] qw[n][k],  m[i] = lo[i] + 2^(n-1) delta[i]
 * (m is the value of centered code 0).  Layouts: x_codes CLQ_CODES_E4M3 with
 * w_codes CLQ_CODES_E4M3 (A4), or x_codes CLQ_CODES_E4M3_SPLIT (A8) with
 * w_codes CLQ_CODES_E4M3 or CLQ_CODES_E4M3_SPLIT; packed operands return
 * CLQ_ERR_UNSUPPORTED.  wsum from clq_weight_code_sums.  acc_dbg receives
 * acc (centered codes).  Other arguments as for clq_linear.
 */
clq_status clq_linear_asym(const uint8_t* Xq, clq_codes x_codes,
                           const float* delta, const float* lo,
                           const uint8_t* W, clq_codes w_codes,
                           const float* s_w, const float* wsum,
                           const void* bias, int32_t M, int32_t N, int32_t K,
                           int32_t b, clq_dtype out_dtype, void* Y,
                           int32_t* acc_dbg, void* stream);

/*
 * Per-layer clip search (Sec. 3.4, Eq. 3, with the layer as its own target
 * layer; Eq. 2's cross-layer target needs a model).  With the symmetric
 * weight grid, l = -r, so the search runs over one percentile p per matrix
 * (the same for every output channel, Sec. 4.1), from host_grid[0 .. G)
 * (values in [0, 1); the paper's range is [beta, gamma] = [0, 0.01]): the
 * clip bound of output channel n is r_n(p) = the floor(p K)-th largest
 * |W~[n][k]| (0-based; p = 0 is the row's absolute maximum, no clipping),
 * W~ = W_p H as in clq_prepare_weights.  For every p the layer runs on the
 * calibration tokens Xcal with the library's own kernels (rotate-quant of
 * Xcal, weights prepared with clip r(p), W4A4 GEMM with bias, output in
 * `dtype`), and host_errors[g] receives sum (Y^ - Yref)^2 over the M x N
 * outputs (fp64, summed in a fixed order).  *host_best receives the index of
 * the smallest error (ties to the smaller index) and clip_out (device fp32
 * [N]) its clip bounds, ready for clq_prepare_weights.
 * W: device [N][ldw], Xcal: device [M][ldx], both of `dtype`; perm: device
 * int32 [K]; Yref: device fp32 [M][N], the layer's full-precision output
 * (X W^T + bias) computed by the caller; bias: device [N] of `dtype` or
 * NULL.  workspace: device, 256-byte aligned, at least
 * clq_clip_search_workspace_size(M, N, K, host_grid, G) bytes.  Offline: the
 * call SYNCHRONIZES `stream` to read the errors back.
 */
size_t clq_clip_search_workspace_size(int32_t M, int32_t N, int32_t K,
                                      const float* host_grid, int32_t G);
clq_status clq_clip_search(const void* W, clq_dtype dtype, int32_t N, int32_t K,
                           int32_t ldw, const int32_t* perm, int32_t b,
                           const void* Xcal, int32_t M, int32_t ldx,
                           const float* Yref, const void* bias,
                           const float* host_grid, int32_t G, float* clip_out,
                           double* host_errors, int32_t* host_best,
                           void* workspace, size_t workspace_bytes,
                           void* stream);

/*
 * Bytes of device workspace clq_fused_linear needs for M tokens of K
 * channels (E4M3 activation codes, scales and per-tile readiness counters).
 */
size_t clq_fused_linear_workspace_size(int32_t M, int32_t K);

/*
 * The whole layer in one persistent kernel: every CTA rotates and quantizes
 * token rows into `workspace` (which stays in L2 for the layer sizes of the
 * paper's models) and runs GEMM tiles, each of which starts as soon as the
 * rows of its token block are published.  With E4M3 weights and K <= 9216
 * the two run side by side in every CTA; otherwise each CTA first finishes
 * its rows, then turns to the GEMM.  Same
 * arithmetic and results as clq_rotate_quant_act followed by
 * clq_w4a4_linear.  X: device [M][ldx] of `dtype`; Y: device [M][N] of
 * `dtype`; bias: device [N] of `dtype` or NULL; W / w_codes: weights in any
 * 4-bit layout, as for clq_w4a4_linear (the activation codes in the
 * workspace then take E2M3 beside E2M3 weights, else E4M3); workspace:
 * device, 256-byte aligned, at least
 * clq_fused_linear_workspace_size(M, K) bytes, owned by the caller and
 * overwritten by the call.
 */
clq_status clq_fused_linear(const void* X, clq_dtype dtype, int32_t M,
                            int32_t K, int32_t ldx, const int32_t* perm,
                            int32_t b, const uint8_t* W, clq_codes w_codes,
                            const float* s_w, const void* bias, int32_t N,
                            void* Y, void* workspace, size_t workspace_bytes,
                            void* stream);

/*
 * Scratch-free variant of clq_fused_linear.  The paper has no counterpart;
 * this entry point exists for callers that cannot allocate device memory
 * where they run the layer: plugin enqueue hooks of inference engines,
 * serving loops that forbid allocation once started, code that holds no
 * allocator.  It takes no workspace.  Instead it uses one scratch array of
 * CLQ_NOALLOC_SCRATCH_BYTES bytes that the library defines in static device
 * memory; every GPU that loads the library holds that array until the
 * process exits.  The call allocates and frees nothing and otherwise behaves
 * exactly like clq_fused_linear (same arguments minus the workspace, same
 * results).
 *  - Problems whose clq_fused_linear_workspace_size(M, K) exceeds
 *    CLQ_NOALLOC_SCRATCH_BYTES are rejected with CLQ_ERR_SCRATCH_LIMIT and
 *    nothing is launched.
 *  - The first call on a device looks up the array's device address
 *    (cudaGetSymbolAddress); make that first call before any stream capture.
 *  - All calls on a device share the one array.  Each call resets the
 *    counters it needs before its kernel runs, but leaves the codes of the
 *    previous call in place; calls whose kernels may overlap on the GPU
 *    (unordered streams) race on the array and must not be issued.
 */
#define CLQ_NOALLOC_SCRATCH_BYTES (64u << 20) /* 64 MiB */
clq_status clq_fused_linear_noalloc(const void* X, clq_dtype dtype, int32_t M,
                                    int32_t K, int32_t ldx,
                                    const int32_t* perm, int32_t b,
                                    const uint8_t* W, clq_codes w_codes,
                                    const float* s_w, const void* bias,
                                    int32_t N, void* Y, void* stream);

/*
 * Synchronize `stream`, then read and clear the device status word of the
 * current device: *out receives CLQ_OK or the first device-side error
 * recorded since the last read.
 */
clq_status clq_get_device_status(void* stream, int32_t* out);

/*
 * Self-test of the bounded-wait machinery: launches one CTA that waits on an
 * mbarrier nothing will ever complete, with a limit of timeout_ns
 * nanoseconds (1e3 .. 1e9).  The wait must give up, record CLQ_ERR_TIMEOUT
 * in the device status word and return, leaving the context usable.
 */
clq_status clq_selftest_bounded_wait(int64_t timeout_ns, void* stream);

/*
 * Peak-rate microbenchmarks (measurement only; the paper has no counterpart:
 * they give the measured denominators next to the GEMM and rotate-quant
 * rates).  Each call launches on `stream` and returns at once; the caller
 * times the launch with CUDA events on that stream and divides *ops by the
 * elapsed time.  *ops receives the multiply-accumulates (or bytes) the
 * launch performs.  No inputs are read except `buf`.
 *
 * clq_peak_tcgen05_e4m3: tcgen05.mma kind::f8f6f4 (E4M3 x E4M3, fp32
 *   accumulate, the MMA of clq_w4a4_linear), one CTA per SM issuing `iters`
 *   K = 128 steps of 128 x 256 tiles from shared memory (1 .. 1e6).
 * clq_peak_mma_sync: warp-level mma.sync, kind 0 = s8 m16n8k32 (the INT8
 *   tensor path of sm_103a), 1 = s4 m16n8k64, 2 = e4m3 m16n8k32; `iters`
 *   (1 .. 1e6) rounds of 4 independent MMAs per warp, 32 warps per SM.
 * clq_peak_hbm_read: reads `bytes` (a multiple of 16, buf 16-byte aligned)
 *   once; *ops = bytes.
 * clq_peak_operand_stream: the W4A4 GEMM's main loop without its epilogue,
 *   one CTA per SM walking `tiles` (1 .. 1e5) 128 x 256 output tiles of
 *   K / 128 steps: a TMA producer fills a ring of four stages with the
 *   GEMM's operand boxes (A 128 rows, B 256 rows, 128 codes a row, 48 KB of
 *   shared memory a step in either layout) taken from `buf`, a device code
 *   array of `rows` x K codes in layout `codes` (CLQ_CODES_E4M3 or
 *   CLQ_CODES_E2M3; rows a multiple of 256, K a multiple of 128, buf 32-byte
 *   aligned).  mma = 0: each stage is released as soon as it lands, *ops =
 *   the shared-memory bytes filled (the rate an SM takes operands in);
 *   mma = 1: the GEMM's four 128 x 256 x 32 MMAs run on each stage, *ops =
 *   the multiply-accumulates.
 * clq_peak_rq_stream: the memory side of clq_rotate_quant_act's b = 64 loop
 *   alone, on X (device [M][K] 16-bit values, rows contiguous): the loop's
 *   tiles, two-stage bulk-copy ring, threads per CTA and programmatic-launch
 *   prologue, writing 1 byte per element to Q (device [M][K]: the high byte
 *   of each value) and 4 bytes per row to S (device fp32 [M]), with no
 *   gather and no arithmetic.  *ops = the rotate-quant algorithmic bytes of
 *   the shape, M (2.5 K + 4), so that ops / time compares with the kernel's
 *   own rate.  Requires M >= 1, 64 <= K <= 16384, K % 64 == 0; X and Q
 *   16-byte aligned.
 */
clq_status clq_peak_tcgen05_e4m3(int32_t iters, int64_t* ops, void* stream);
clq_status clq_peak_mma_sync(int32_t kind, int32_t iters, int64_t* ops, void* stream);
clq_status clq_peak_hbm_read(const void* buf, uint64_t bytes, int64_t* ops, void* stream);
clq_status clq_peak_operand_stream(const uint8_t* buf, int32_t rows, int32_t K,
                                   clq_codes codes, int32_t mma, int32_t tiles,
                                   int64_t* ops, void* stream);
clq_status clq_peak_rq_stream(const void* X, int32_t M, int32_t K, uint8_t* Q, float* S,
                              int64_t* ops, void* stream);

#ifdef __cplusplus
}
#endif

#endif /* CLQ_H */
