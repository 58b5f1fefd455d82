"""Python binding of libclq (include/clq.h): argument marshalling only.

Two layers:

* ``clq_*`` functions with the C names and C arguments (integers for device
  pointers and the stream), returning the status code;
* tensor helpers (``rotate_quant_act``, ``w4a4_linear`` ...) that take torch
  tensors, allocate outputs with torch, pass their pointers and the current
  stream to the C call, and raise ``ClqError`` on a non-zero status.

Every step of the computation runs in the CUDA kernels of libclq.so; there is
no CPU or PyTorch fallback.  If the library is missing, the first call raises.
"""
import ctypes
import os

import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libclq.so")

CLQ_F16, CLQ_BF16 = 0, 1
CLQ_CODES_INT4_PACKED, CLQ_CODES_E4M3, CLQ_CODES_E4M3_SPLIT, CLQ_CODES_E2M3 = 0, 1, 2, 3
STATUS = {0: "CLQ_OK", 1: "CLQ_ERR_INVALID_ARG", 2: "CLQ_ERR_SHAPE",
          3: "CLQ_ERR_ALIGN", 4: "CLQ_ERR_UNSUPPORTED", 5: "CLQ_ERR_CUDA",
          6: "CLQ_ERR_TIMEOUT", 7: "CLQ_ERR_DEVICE_INDEX",
          8: "CLQ_ERR_SCRATCH_LIMIT", 9: "CLQ_ERR_DEVICE_CODE"}
EXPORTS = ("clq_status_string", "clq_version", "clq_outlier_scores",
           "clq_build_permutation", "clq_prepare_weights",
           "clq_rotate_quant_act", "clq_expand_weights", "clq_w4a4_linear",
           "clq_fused_linear_workspace_size", "clq_fused_linear",
           "clq_fused_linear_noalloc", "clq_get_device_status",
           "clq_selftest_bounded_wait", "clq_outlier_scores_metric",
           "clq_peak_tcgen05_e4m3",
           "clq_peak_mma_sync", "clq_peak_hbm_read",
           "clq_prepare_weights_codes", "clq_linear",
           "clq_rotate_quant_act_asym", "clq_weight_code_sums",
           "clq_linear_asym", "clq_clip_search_workspace_size",
           "clq_clip_search", "clq_convert_codes", "clq_peak_operand_stream",
           "clq_peak_rq_stream")

_lib = None
_P = ctypes.c_void_p
_I = ctypes.c_int32
_Z = ctypes.c_size_t
_SIGS = {
    "clq_status_string": (ctypes.c_char_p, [_I]),
    "clq_version": (_I, []),
    "clq_outlier_scores": (_I, [_P, _I, _I, _I, _I, _P, _P]),
    "clq_outlier_scores_metric": (_I, [_P, _I, _I, _I, _I, _I, _P, _P]),
    "clq_build_permutation": (_I, [_P, _I, _P]),
    "clq_prepare_weights": (_I, [_P, _I, _I, _I, _I, _P, _I, _P, _P, _P, _P,
                                 _P]),
    "clq_rotate_quant_act": (_I, [_P, _I, _I, _I, _I, _P, _I, _I, _P, _P, _P,
                                  _P]),
    "clq_expand_weights": (_I, [_P, _I, _I, _P, _P]),
    "clq_convert_codes": (_I, [_P, _I, _P, _I, _I, _I, _P]),
    "clq_w4a4_linear": (_I, [_P, _I, _P, _P, _I, _P, _P, _I, _I, _I, _I, _I,
                             _P, _P, _P]),
    "clq_fused_linear_workspace_size": (_Z, [_I, _I]),
    "clq_fused_linear": (_I, [_P, _I, _I, _I, _I, _P, _I, _P, _I, _P, _P, _I,
                              _P, _P, _Z, _P]),
    "clq_fused_linear_noalloc": (_I, [_P, _I, _I, _I, _I, _P, _I, _P, _I, _P,
                                      _P, _I, _P, _P]),
    "clq_get_device_status": (_I, [_P, _P]),
    "clq_selftest_bounded_wait": (_I, [ctypes.c_int64, _P]),
    "clq_peak_tcgen05_e4m3": (_I, [_I, _P, _P]),
    "clq_peak_mma_sync": (_I, [_I, _I, _P, _P]),
    "clq_peak_hbm_read": (_I, [_P, ctypes.c_uint64, _P, _P]),
    "clq_peak_operand_stream": (_I, [_P, _I, _I, _I, _I, _I, _P, _P]),
    "clq_peak_rq_stream": (_I, [_P, _I, _I, _P, _P, _P, _P]),
    "clq_prepare_weights_codes": (_I, [_P, _I, _I, _I, _I, _P, _I, _P, _I,
                                       _P, _P, _P, _P]),
    "clq_linear": (_I, [_P, _I, _P, _P, _I, _P, _P, _I, _I, _I, _I, _I, _P,
                        _P, _P]),
    "clq_rotate_quant_act_asym": (_I, [_P, _I, _I, _I, _I, _P, _I, _I, _P,
                                       _P, _P, _P, _P]),
    "clq_weight_code_sums": (_I, [_P, _I, _I, _I, _P, _P]),
    "clq_linear_asym": (_I, [_P, _I, _P, _P, _P, _I, _P, _P, _P, _I, _I, _I,
                             _I, _I, _P, _P, _P]),
    "clq_clip_search_workspace_size": (_Z, [_I, _I, _I, _P, _I]),
    "clq_clip_search": (_I, [_P, _I, _I, _I, _I, _P, _I, _P, _I, _I, _P, _P,
                             _P, _I, _P, _P, _P, _P, _Z, _P]),
}


class ClqError(RuntimeError):
    def __init__(self, status, where):
        self.status = int(status)
        super().__init__("%s failed: %s" % (where, status_string(status)))


def load():
    """Load libclq.so (built in-tree by ``build.build()``)."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError("libclq.so is not built (%s); run "
                               "paper_2509_24416_gb300.build.build()"
                               % LIB_PATH)
        lib = ctypes.CDLL(LIB_PATH)
        for name, (res, args) in _SIGS.items():
            fn = getattr(lib, name)
            fn.restype = res
            fn.argtypes = args
        _lib = lib
    return _lib


def status_string(status):
    try:
        return load().clq_status_string(int(status)).decode()
    except RuntimeError:
        return STATUS.get(int(status), "unknown")


# ------------------------------------------------- C-named raw entry points --
def clq_outlier_scores(calib, dtype, B, T, K, scores, stream):
    return load().clq_outlier_scores(calib, dtype, B, T, K, scores, stream)


def clq_build_permutation(host_scores, K, host_perm):
    return load().clq_build_permutation(host_scores, K, host_perm)


def clq_prepare_weights(W, dtype, N, K, ldw, perm, b, clip, Wq, s_w,
                        w_rot_dbg, stream):
    return load().clq_prepare_weights(W, dtype, N, K, ldw, perm, b, clip, Wq,
                                      s_w, w_rot_dbg, stream)


def clq_prepare_weights_codes(W, dtype, N, K, ldw, perm, b, clip, w_codes,
                              Wq, s_w, w_rot_dbg, stream):
    return load().clq_prepare_weights_codes(W, dtype, N, K, ldw, perm, b,
                                            clip, w_codes, Wq, s_w, w_rot_dbg,
                                            stream)


def clq_linear(Xq, x_codes, s_x, W, w_codes, s_w, bias, M, N, K, b,
               out_dtype, Y, acc_dbg, stream):
    return load().clq_linear(Xq, x_codes, s_x, W, w_codes, s_w, bias, M, N,
                             K, b, out_dtype, Y, acc_dbg, stream)


def clq_rotate_quant_act_asym(X, dtype, M, K, ldx, perm, b, x_codes, Xq, delta,
                              lo, x_rot_dbg, stream):
    return load().clq_rotate_quant_act_asym(X, dtype, M, K, ldx, perm, b,
                                            x_codes, Xq, delta, lo, x_rot_dbg,
                                            stream)


def clq_weight_code_sums(W, w_codes, N, K, wsum, stream):
    return load().clq_weight_code_sums(W, w_codes, N, K, wsum, stream)


def clq_linear_asym(Xq, x_codes, delta, lo, W, w_codes, s_w, wsum, bias, M, N,
                    K, b, out_dtype, Y, acc_dbg, stream):
    return load().clq_linear_asym(Xq, x_codes, delta, lo, W, w_codes, s_w, wsum,
                                  bias, M, N, K, b, out_dtype, Y, acc_dbg,
                                  stream)


def clq_clip_search_workspace_size(M, N, K, host_grid, G):
    return load().clq_clip_search_workspace_size(M, N, K, host_grid, G)


def clq_clip_search(W, dtype, N, K, ldw, perm, b, Xcal, M, ldx, Yref, bias,
                    host_grid, G, clip_out, host_errors, host_best, workspace,
                    workspace_bytes, stream):
    return load().clq_clip_search(W, dtype, N, K, ldw, perm, b, Xcal, M, ldx,
                                  Yref, bias, host_grid, G, clip_out,
                                  host_errors, host_best, workspace,
                                  workspace_bytes, stream)


def clq_rotate_quant_act(X, dtype, M, K, ldx, perm, b, x_codes, Xq, s_x,
                         x_rot_dbg, stream):
    return load().clq_rotate_quant_act(X, dtype, M, K, ldx, perm, b, x_codes,
                                       Xq, s_x, x_rot_dbg, stream)


def clq_expand_weights(Wq, N, K, We, stream):
    return load().clq_expand_weights(Wq, N, K, We, stream)


def clq_convert_codes(src, src_codes, dst, dst_codes, rows, K, stream):
    return load().clq_convert_codes(src, src_codes, dst, dst_codes, rows, K, stream)


def clq_w4a4_linear(Xq, x_codes, s_x, W, w_codes, s_w, bias, M, N, K, b,
                    out_dtype, Y, acc_dbg, stream):
    return load().clq_w4a4_linear(Xq, x_codes, s_x, W, w_codes, s_w, bias, M,
                                  N, K, b, out_dtype, Y, acc_dbg, stream)


def clq_fused_linear_workspace_size(M, K):
    return load().clq_fused_linear_workspace_size(M, K)


def clq_fused_linear(X, dtype, M, K, ldx, perm, b, W, w_codes, s_w, bias, N,
                     Y, workspace, workspace_bytes, stream):
    return load().clq_fused_linear(X, dtype, M, K, ldx, perm, b, W, w_codes,
                                   s_w, bias, N, Y, workspace,
                                   workspace_bytes, stream)


def clq_fused_linear_noalloc(X, dtype, M, K, ldx, perm, b, W, w_codes, s_w,
                             bias, N, Y, stream):
    return load().clq_fused_linear_noalloc(X, dtype, M, K, ldx, perm, b, W,
                                           w_codes, s_w, bias, N, Y, stream)


def clq_get_device_status(stream, out):
    return load().clq_get_device_status(stream, out)


def clq_selftest_bounded_wait(timeout_ns, stream):
    return load().clq_selftest_bounded_wait(timeout_ns, stream)


def clq_outlier_scores_metric(calib, dtype, B, T, K, metric, scores, stream):
    return load().clq_outlier_scores_metric(calib, dtype, B, T, K, metric, scores, stream)


def clq_peak_tcgen05_e4m3(iters, ops, stream):
    return load().clq_peak_tcgen05_e4m3(iters, ops, stream)


def clq_peak_mma_sync(kind, iters, ops, stream):
    return load().clq_peak_mma_sync(kind, iters, ops, stream)


def clq_peak_rq_stream(X, M, K, Q, S, ops, stream):
    return load().clq_peak_rq_stream(X, M, K, Q, S, ops, stream)


def clq_peak_operand_stream(buf, rows, K, codes, mma, tiles, ops, stream):
    return load().clq_peak_operand_stream(buf, rows, K, codes, mma, tiles, ops, stream)


def clq_peak_hbm_read(buf, nbytes, ops, stream):
    return load().clq_peak_hbm_read(buf, nbytes, ops, stream)


# ----------------------------------------------------------- tensor helpers --
def _dt(t):
    if t.dtype == torch.float16:
        return CLQ_F16
    if t.dtype == torch.bfloat16:
        return CLQ_BF16
    raise TypeError("expected float16 or bfloat16, got %s" % t.dtype)


def _ptr(t):
    return None if t is None else t.data_ptr()


def _stream(stream):
    s = torch.cuda.current_stream() if stream is None else stream
    return s.cuda_stream


def _check(st, where):
    if st != 0:
        raise ClqError(st, where)


def _buffer(t, shape, dtype, device, name):
    """A caller-provided output buffer, checked against what the call will
    write (the C ABI takes plain pointers and cannot check sizes)."""
    if tuple(t.shape) != tuple(shape) or t.dtype != dtype or not t.is_contiguous():
        raise ValueError("%s must be a contiguous %s tensor of shape %s, got %s %s"
                         % (name, dtype, tuple(shape), t.dtype, tuple(t.shape)))
    if t.device != torch.device(device):
        raise ValueError("%s must be on %s" % (name, device))
    return t


def _row_major(t, name):
    if t.dim() != 2 or t.stride(1) != 1:
        raise ValueError("%s must be a 2-D tensor with unit column stride"
                         % name)


OUTLIER_METRICS = {"absmax": 0, "percentile": 1, "topk_mean": 2, "range": 3, "par": 4}


def outlier_scores(calib, metric="absmax", stream=None):
    """calib [B, T, K] fp16/bf16 on the GPU -> fp32 scores [K] under `metric`
    (one of OUTLIER_METRICS; "absmax" is the method's, Sec. 3.3)."""
    calib = calib.contiguous()
    B, T, K = calib.shape
    scores = torch.empty(K, dtype=torch.float32, device=calib.device)
    if metric == "absmax":
        _check(clq_outlier_scores(_ptr(calib), _dt(calib), B, T, K, _ptr(scores),
                                  _stream(stream)), "clq_outlier_scores")
    else:
        if metric not in OUTLIER_METRICS:
            raise ValueError("unknown outlier metric %r" % (metric,))
        _check(clq_outlier_scores_metric(_ptr(calib), _dt(calib), B, T, K,
                                         OUTLIER_METRICS[metric], _ptr(scores),
                                         _stream(stream)), "clq_outlier_scores_metric")
    return scores


def build_permutation(scores):
    """Host column-swap vector from scores (any device) -> int32 CPU [K]."""
    s = scores.detach().to("cpu", torch.float32).contiguous()
    K = s.numel()
    perm = torch.empty(K, dtype=torch.int32)
    _check(clq_build_permutation(_ptr(s), K, _ptr(perm)),
           "clq_build_permutation")
    return perm


def codes_width(codes, K):
    """Bytes per row of K codes in layout `codes`."""
    return {CLQ_CODES_INT4_PACKED: K // 2, CLQ_CODES_E4M3: K,
            CLQ_CODES_E4M3_SPLIT: 2 * K, CLQ_CODES_E2M3: K // 4 * 3}[codes]


def exec_layout(K):
    """The default 4-bit execution layout for K input channels: E4M3, one
    byte a code, the layout the W4A4 step runs fastest with (measured: the
    GEMM's TMA fills shared memory with the same padded bytes for E2M3, and
    its 16-code groups cost the rotate-quant store extra work).  E2M3
    (0.75 B a code, K % 128 == 0) is the layout to pass as ``w_codes`` when
    resident weight memory matters more."""
    return CLQ_CODES_E4M3


def prepare_weights(W, perm, b, clip=None, with_rot=False, stream=None,
                    codes=CLQ_CODES_INT4_PACKED):
    """W [N, K] -> (Wq uint8 [N, width], s_w fp32 [N][, w_rot fp32 [N, K]]);
    4-bit codes packed ([N, K/2], the default) or E4M3 ([N, K]), or 8-bit
    codes as split planes ([N, 2K], CLQ_CODES_E4M3_SPLIT)."""
    _row_major(W, "W")
    N, K = W.shape
    dev = W.device
    Wq = torch.empty((N, codes_width(codes, K)), dtype=torch.uint8, device=dev)
    s_w = torch.empty(N, dtype=torch.float32, device=dev)
    rot = (torch.empty((N, K), dtype=torch.float32, device=dev)
           if with_rot else None)
    if codes == CLQ_CODES_INT4_PACKED:
        _check(clq_prepare_weights(_ptr(W), _dt(W), N, K, W.stride(0),
                                   _ptr(perm), b, _ptr(clip), _ptr(Wq),
                                   _ptr(s_w), _ptr(rot), _stream(stream)),
               "clq_prepare_weights")
    else:
        _check(clq_prepare_weights_codes(_ptr(W), _dt(W), N, K, W.stride(0),
                                         _ptr(perm), b, _ptr(clip), codes,
                                         _ptr(Wq), _ptr(s_w), _ptr(rot),
                                         _stream(stream)),
               "clq_prepare_weights_codes")
    return (Wq, s_w, rot) if with_rot else (Wq, s_w)


def rotate_quant_act(X, perm, b, codes=CLQ_CODES_INT4_PACKED, Xq=None, s_x=None,
                     with_rot=False, stream=None):
    """X [M, K] -> (Xq uint8, s_x fp32 [M][, x_rot fp32 [M, K]]); Xq is
    [M, K/2] packed (CLQ_CODES_INT4_PACKED), [M, K] E4M3 (CLQ_CODES_E4M3) or,
    for 8-bit codes, [M, 2K] split planes (CLQ_CODES_E4M3_SPLIT)."""
    _row_major(X, "X")
    M, K = X.shape
    dev = X.device
    if Xq is None:
        Xq = torch.empty((M, codes_width(codes, K)), dtype=torch.uint8,
                         device=dev)
    else:
        _buffer(Xq, (M, codes_width(codes, K)), torch.uint8, dev, "Xq")
    if s_x is None:
        s_x = torch.empty(M, dtype=torch.float32, device=dev)
    else:
        _buffer(s_x, (M,), torch.float32, dev, "s_x")
    rot = (torch.empty((M, K), dtype=torch.float32, device=dev)
           if with_rot else None)
    _check(clq_rotate_quant_act(_ptr(X), _dt(X), M, K, X.stride(0),
                                _ptr(perm), b, codes, _ptr(Xq), _ptr(s_x),
                                _ptr(rot), _stream(stream)),
           "clq_rotate_quant_act")
    return (Xq, s_x, rot) if with_rot else (Xq, s_x)


def rotate_quant_act_asym(X, perm, b, codes=CLQ_CODES_E4M3, Xq=None,
                          delta=None, lo=None, with_rot=False, stream=None):
    """X [M, K] -> (Xq uint8, delta fp32 [M], lo fp32 [M][, x_rot fp32
    [M, K]]): asymmetric codes (Eq. 1, dynamic min / max) stored centered,
    4-bit in CLQ_CODES_E4M3 / CLQ_CODES_INT4_PACKED, 8-bit in
    CLQ_CODES_E4M3_SPLIT."""
    _row_major(X, "X")
    M, K = X.shape
    dev = X.device
    if Xq is None:
        Xq = torch.empty((M, codes_width(codes, K)), dtype=torch.uint8,
                         device=dev)
    else:
        _buffer(Xq, (M, codes_width(codes, K)), torch.uint8, dev, "Xq")
    if delta is None:
        delta = torch.empty(M, dtype=torch.float32, device=dev)
    else:
        _buffer(delta, (M,), torch.float32, dev, "delta")
    if lo is None:
        lo = torch.empty(M, dtype=torch.float32, device=dev)
    else:
        _buffer(lo, (M,), torch.float32, dev, "lo")
    rot = (torch.empty((M, K), dtype=torch.float32, device=dev)
           if with_rot else None)
    _check(clq_rotate_quant_act_asym(_ptr(X), _dt(X), M, K, X.stride(0),
                                     _ptr(perm), b, codes, _ptr(Xq),
                                     _ptr(delta), _ptr(lo), _ptr(rot),
                                     _stream(stream)),
           "clq_rotate_quant_act_asym")
    return (Xq, delta, lo, rot) if with_rot else (Xq, delta, lo)


def weight_code_sums(W, K, stream=None):
    """Integer code sums of each row of a weight code array (any layout) ->
    fp32 [N]."""
    N = W.shape[0]
    wsum = torch.empty(N, dtype=torch.float32, device=W.device)
    _check(clq_weight_code_sums(_ptr(W), codes_layout(W, K), N, K, _ptr(wsum),
                                _stream(stream)), "clq_weight_code_sums")
    return wsum


def expand_weights(Wq, stream=None):
    """Packed codes [N, K/2] -> E4M3 execution layout [N, K] (uint8)."""
    N, Kh = Wq.shape
    We = torch.empty((N, 2 * Kh), dtype=torch.uint8, device=Wq.device)
    _check(clq_expand_weights(_ptr(Wq), N, 2 * Kh, _ptr(We), _stream(stream)),
           "clq_expand_weights")
    return We


def codes_layout(t, K):
    """Layout of a code array of K codes per row, from its width."""
    if t.shape[1] == K:
        return CLQ_CODES_E4M3
    if 2 * t.shape[1] == K:
        return CLQ_CODES_INT4_PACKED
    if t.shape[1] == 2 * K:
        return CLQ_CODES_E4M3_SPLIT
    if 4 * t.shape[1] == 3 * K:
        return CLQ_CODES_E2M3
    raise ValueError("codes must be [rows, K/2] packed, [rows, K] E4M3, "
                     "[rows, 3K/4] E2M3 or [rows, 2K] split")


def convert_codes(src, K, dst_codes, dst=None, stream=None):
    """A 4-bit code array in any layout -> the same codes in layout
    `dst_codes` (uint8 [rows, width])."""
    rows = src.shape[0]
    width = codes_width(dst_codes, K)
    if dst is None:
        dst = torch.empty((rows, width), dtype=torch.uint8, device=src.device)
    else:
        _buffer(dst, (rows, width), torch.uint8, src.device, "dst")
    _check(clq_convert_codes(_ptr(src), codes_layout(src, K), _ptr(dst), dst_codes,
                             rows, K, _stream(stream)), "clq_convert_codes")
    return dst


def w4a4_linear(Xq, s_x, W, s_w, b, K, bias=None, out_dtype=torch.float16,
                Y=None, with_acc=False, stream=None):
    """Activation codes x weight codes (each packed [rows, K/2] or E4M3
    [rows, K]) -> Y [M, N] (out_dtype)[, acc int32 [M, N]]."""
    M = Xq.shape[0]
    N = W.shape[0]
    if Y is None:
        Y = torch.empty((M, N), dtype=out_dtype, device=Xq.device)
    else:
        _buffer(Y, (M, N), Y.dtype, Xq.device, "Y")
    acc = (torch.empty((M, N), dtype=torch.int32, device=Xq.device)
           if with_acc else None)
    if bias is not None and bias.dtype != Y.dtype:
        raise TypeError("bias must have the output dtype")
    _check(clq_w4a4_linear(_ptr(Xq), codes_layout(Xq, K), _ptr(s_x), _ptr(W),
                           codes_layout(W, K), _ptr(s_w), _ptr(bias), M, N, K,
                           b, _dt(Y), _ptr(Y), _ptr(acc), _stream(stream)),
           "clq_w4a4_linear")
    return (Y, acc) if with_acc else Y


def linear(Xq, s_x, W, s_w, b, K, bias=None, out_dtype=torch.float16,
           Y=None, with_acc=False, stream=None):
    """Codes x codes at any bit setting (W4A4, W4A8, W8A8; layouts inferred
    from the widths) -> Y [M, N] (out_dtype)[, acc int32 [M, N]]."""
    M = Xq.shape[0]
    N = W.shape[0]
    if Y is None:
        Y = torch.empty((M, N), dtype=out_dtype, device=Xq.device)
    else:
        _buffer(Y, (M, N), Y.dtype, Xq.device, "Y")
    acc = (torch.empty((M, N), dtype=torch.int32, device=Xq.device)
           if with_acc else None)
    if bias is not None and bias.dtype != Y.dtype:
        raise TypeError("bias must have the output dtype")
    _check(clq_linear(_ptr(Xq), codes_layout(Xq, K), _ptr(s_x), _ptr(W),
                      codes_layout(W, K), _ptr(s_w), _ptr(bias), M, N, K, b,
                      _dt(Y), _ptr(Y), _ptr(acc), _stream(stream)),
           "clq_linear")
    return (Y, acc) if with_acc else Y


def linear_asym(Xq, delta, lo, W, s_w, wsum, b, K, bias=None,
                out_dtype=torch.float16, Y=None, with_acc=False, stream=None):
    """Asymmetric activation codes (rotate_quant_act_asym) x weight codes
    with the zero-point epilogue -> Y [M, N][, acc int32 [M, N]]."""
    M = Xq.shape[0]
    N = W.shape[0]
    if Y is None:
        Y = torch.empty((M, N), dtype=out_dtype, device=Xq.device)
    else:
        _buffer(Y, (M, N), Y.dtype, Xq.device, "Y")
    acc = (torch.empty((M, N), dtype=torch.int32, device=Xq.device)
           if with_acc else None)
    if bias is not None and bias.dtype != Y.dtype:
        raise TypeError("bias must have the output dtype")
    _check(clq_linear_asym(_ptr(Xq), codes_layout(Xq, K), _ptr(delta), _ptr(lo),
                           _ptr(W), codes_layout(W, K), _ptr(s_w), _ptr(wsum),
                           _ptr(bias), M, N, K, b, _dt(Y), _ptr(Y), _ptr(acc),
                           _stream(stream)), "clq_linear_asym")
    return (Y, acc) if with_acc else Y


CLIP_GRID = tuple(0.001 * i for i in range(11))  # [beta, gamma] = [0, 0.01]


def clip_search(W, perm, b, Xcal, Yref, bias=None, grid=CLIP_GRID, stream=None):
    """Per-layer clip search (Sec. 3.4, Eq. 3): W [N, K], Xcal [M, K] (same
    dtype, on the GPU), Yref fp32 [M, N] the full-precision layer output.
    Returns (clip fp32 [N] of the best percentile, errors fp64 [G] (host),
    best index).  Synchronizes the stream."""
    _row_major(W, "W")
    _row_major(Xcal, "Xcal")
    N, K = W.shape
    M = Xcal.shape[0]
    g32 = torch.tensor(grid, dtype=torch.float32)
    G = g32.numel()
    nbytes = clq_clip_search_workspace_size(M, N, K, _ptr(g32), G)
    if nbytes == 0:
        raise ValueError("invalid clip search shape or grid")
    ws = torch.empty(nbytes, dtype=torch.uint8, device=W.device)
    clip = torch.empty(N, dtype=torch.float32, device=W.device)
    errors = torch.empty(G, dtype=torch.float64)
    best = torch.zeros(1, dtype=torch.int32)
    Yref = Yref.to(torch.float32).contiguous()
    _check(clq_clip_search(_ptr(W), _dt(W), N, K, W.stride(0),
                           _ptr(perm), b, _ptr(Xcal), M, Xcal.stride(0),
                           _ptr(Yref), _ptr(bias), _ptr(g32), G, _ptr(clip),
                           _ptr(errors), _ptr(best), _ptr(ws), nbytes,
                           _stream(stream)), "clq_clip_search")
    return clip, errors, int(best.item())


def fused_workspace(M, K, device):
    """A workspace tensor large enough for fused_linear on M x K inputs."""
    n = clq_fused_linear_workspace_size(M, K)
    return torch.empty(max(n, 256), dtype=torch.uint8, device=device)


def fused_linear(X, perm, b, W, s_w, bias=None, Y=None, workspace=None,
                 stream=None):
    """X [M, K] -> Y [M, N] in X's dtype, rotate-quant and GEMM in one
    kernel.  W is packed [N, K/2], E4M3 [N, K] or E2M3 [N, 3K/4]."""
    _row_major(X, "X")
    M, K = X.shape
    N = W.shape[0]
    if Y is None:
        Y = torch.empty((M, N), dtype=X.dtype, device=X.device)
    else:
        _buffer(Y, (M, N), X.dtype, X.device, "Y")
    if workspace is None:
        workspace = fused_workspace(M, K, X.device)
    _check(clq_fused_linear(_ptr(X), _dt(X), M, K, X.stride(0), _ptr(perm), b,
                            _ptr(W), codes_layout(W, K), _ptr(s_w), _ptr(bias), N,
                            _ptr(Y), _ptr(workspace), workspace.numel(),
                            _stream(stream)), "clq_fused_linear")
    return Y


def device_status(stream=None):
    """Synchronize and read-and-clear the device status word."""
    out = ctypes.c_int32(0)
    _check(clq_get_device_status(_stream(stream), ctypes.addressof(out)),
           "clq_get_device_status")
    return out.value


def selftest_bounded_wait(timeout_ns=1000000, stream=None):
    _check(clq_selftest_bounded_wait(int(timeout_ns), _stream(stream)),
           "clq_selftest_bounded_wait")


class PreparedLinear:
    """A quantized linear layer: the prepared-weight package (codes, s_w,
    perm, b, bias) of Sec. 3.3, where the swap vector is the only stored part
    of G.

    Only one copy of the weight codes is resident on the device, ``We``, in
    the execution layout the GEMM loads directly (``w_codes``): at W4A4 E4M3
    (1 B a weight) by default, or E2M3 (12 bytes per 16 codes, 0.75 B a
    weight, K % 128 == 0) on request; at W4A8 E4M3 (the 8-bit activation
    planes pair with E4M3 weights); at W8A8 the split 8-bit planes.  ``Wq`` gives the
    storage format (packed INT4 nibbles, 4 bits a weight, the format the
    paper's memory figure counts; the split planes at W8A8), converted from
    ``We`` on demand.  Activation codes are produced in an execution layout
    too (they are transient): the 4-bit layout of the weights, or split
    planes for 8-bit activations (a_bits); ``a_codes`` picks another 4-bit
    activation layout (packed nibbles or E4M3 with packed or E4M3 weights,
    E2M3 with E2M3 weights).  ``state_dict()`` keeps the
    storage codes; ``from_state_dict()`` converts them back.  Calling the
    object runs the separate rotate-quant and GEMM kernels (``fused=False``)
    or, at W4A4, the fused kernel.
    """

    def __init__(self, Wq, s_w, perm, b, bias=None, We=None, a_bits=4, w_codes=None,
                 a_codes=None):
        """Wq: weight codes in any layout (packed storage codes, an
        execution layout, or split planes for 8-bit weights); they are
        converted to the execution layout unless ``We`` already holds it."""
        self.s_w, self.perm, self.b, self.bias = s_w, perm, b, bias
        K = perm.numel()
        self.K = K
        src = We if We is not None else Wq
        self.w_bits = 8 if codes_layout(src, K) == CLQ_CODES_E4M3_SPLIT else 4
        if a_bits not in (4, 8) or (self.w_bits == 8 and a_bits != 8):
            raise ValueError("bit settings are W4A4, W4A8 and W8A8")
        self.a_bits = a_bits
        if self.w_bits == 8:
            self.w_codes = CLQ_CODES_E4M3_SPLIT
        elif w_codes is not None:
            self.w_codes = w_codes
        else:
            self.w_codes = exec_layout(K) if a_bits == 4 else CLQ_CODES_E4M3
        if codes_layout(src, K) == self.w_codes:
            self.We = src
        else:
            self.We = convert_codes(src, K, self.w_codes)
        if a_codes is not None:
            four = (CLQ_CODES_INT4_PACKED, CLQ_CODES_E4M3, CLQ_CODES_E2M3)
            if a_bits != 4 or a_codes not in four or self.w_codes not in four or (
                    (a_codes == CLQ_CODES_E2M3) != (self.w_codes == CLQ_CODES_E2M3)):
                raise ValueError("4-bit activation codes pair packed or E4M3 with packed "
                                 "or E4M3 weights, and E2M3 with E2M3")
        self._a_codes = a_codes

    @property
    def Wq(self):
        """Storage codes: packed INT4 nibbles [N, K/2] (4-bit weights), or the
        split planes [N, 2K] (8-bit weights), converted from ``We``."""
        if self.w_bits == 8:
            return self.We
        if self.w_codes == CLQ_CODES_INT4_PACKED:
            return self.We
        return convert_codes(self.We, self.K, CLQ_CODES_INT4_PACKED)

    def resident_bytes(self):
        """Device bytes the layer keeps: weight codes, scales, swap vector,
        bias."""
        n = self.We.numel() + self.s_w.numel() * 4 + self.perm.numel() * 4
        if self.bias is not None:
            n += self.bias.numel() * self.bias.element_size()
        return n

    @classmethod
    def from_weight(cls, W, perm, b, bias=None, clip=None, a_bits=4, w_bits=4,
                    w_codes=None, a_codes=None):
        perm = perm.to(W.device, torch.int32).contiguous()
        K = W.shape[1]
        if w_bits == 8:
            codes = CLQ_CODES_E4M3_SPLIT
        elif w_codes is not None:
            codes = w_codes
        else:
            codes = exec_layout(K) if a_bits == 4 else CLQ_CODES_E4M3
        We, s_w = prepare_weights(W.contiguous(), perm, b, clip, codes=codes)
        return cls(None, s_w, perm, b, bias, We=We, a_bits=a_bits, w_codes=codes,
                   a_codes=a_codes)

    @classmethod
    def calibrate(cls, W, calib, b, bias=None, metric="absmax", clip_grid=None,
                  a_bits=4, w_bits=4, stream=None):
        """The offline steps in the paper's order (Sec. 3.3, Sec. 3.4), all on
        the GPU: outlier scores of the calibration batch calib [B, T, K]
        under `metric` (Sec. 4.4 names the alternatives), the swap vector,
        then, when `clip_grid` is given (e.g. CLIP_GRID) and the weights are
        4-bit, the per-layer clip search (Eq. 3) on the B * T calibration
        tokens against their fp32 product, and finally the prepared layer.
        Returns (layer, info) with info = dict(scores, perm, clip, errors,
        best)."""
        K = W.shape[1]
        scores = outlier_scores(calib, metric=metric, stream=stream)
        perm = build_permutation(scores).to(W.device)
        clip = errors = best = None
        if clip_grid is not None and w_bits == 4:
            Xcal = calib.reshape(-1, K).contiguous()
            # The search's target, the layer's full-precision output: taken in
            # fp64 and rounded once to fp32, so that no matmul setting of the
            # caller (TF32, reduced-precision reductions) changes the objective.
            Yref = Xcal.double() @ W.double().t()
            if bias is not None:
                Yref = Yref + bias.double()[None, :]
            Yref = Yref.float().contiguous()
            clip, errors, best = clip_search(W.contiguous(), perm, b, Xcal, Yref, bias,
                                             grid=clip_grid, stream=stream)
        layer = cls.from_weight(W, perm, b, bias=bias, clip=clip, a_bits=a_bits,
                                w_bits=w_bits)
        return layer, dict(scores=scores, perm=perm, clip=clip, errors=errors, best=best)

    @property
    def act_codes(self):
        """Layout of the activation codes the separate path writes: split
        planes for 8-bit activations, else the ``a_codes`` given, else the
        4-bit layout of the weights (E2M3 with E2M3, E4M3 otherwise)."""
        if self.a_bits == 8:
            return CLQ_CODES_E4M3_SPLIT
        if self._a_codes is not None:
            return self._a_codes
        return CLQ_CODES_E2M3 if self.w_codes == CLQ_CODES_E2M3 else CLQ_CODES_E4M3

    def state_dict(self):
        d = dict(Wq=self.Wq, s_w=self.s_w, perm=self.perm,
                 b=torch.tensor(self.b), a_bits=torch.tensor(self.a_bits))
        if self.bias is not None:
            d["bias"] = self.bias
        return d

    @classmethod
    def from_state_dict(cls, d):
        a_bits = int(d["a_bits"]) if "a_bits" in d else 4
        return cls(d["Wq"], d["s_w"], d["perm"], int(d["b"]), d.get("bias"),
                   a_bits=a_bits)

    def __call__(self, X, fused=False, workspace=None, stream=None, Y=None,
                 Xq=None, s_x=None):
        """Y = X W^T + bias at the layer's bit setting.  Y, and the activation
        codes / scales of the separate path (Xq [M, K] uint8 for 4-bit, [M, 2K]
        for 8-bit activations; s_x [M] fp32), may be passed in to avoid
        allocations."""
        if fused:
            if self.a_bits != 4:
                raise ValueError("the fused kernel runs W4A4 only")
            return fused_linear(X, self.perm, self.b, self.We, self.s_w,
                                self.bias, Y=Y, workspace=workspace, stream=stream)
        codes = self.act_codes
        Xq, s_x = rotate_quant_act(X, self.perm, self.b, codes,
                                   Xq=Xq, s_x=s_x, stream=stream)
        if self.a_bits == 4:
            return w4a4_linear(Xq, s_x, self.We, self.s_w, self.b, X.shape[1],
                               self.bias, out_dtype=X.dtype, Y=Y, stream=stream)
        return linear(Xq, s_x, self.We, self.s_w, self.b, X.shape[1],
                      self.bias, out_dtype=X.dtype, Y=Y, stream=stream)


class HostPipeline:
    """Runs prepared layers on host inputs into host outputs with the three
    kinds of work on three CUDA streams, so that they overlap: while layer i
    computes, layer i + 1's input travels to the device and layer i - 1's
    output travels back.  All device buffers (inputs, codes, scales,
    workspaces, outputs) are allocated once here; host buffers should be
    pinned (`torch.Tensor.pin_memory`) for the copies to be asynchronous.

    `layers` is a list of (PreparedLinear, M, K, N).  `run` enqueues one pass
    and returns at once; a later `run` waits on the device, per layer, for the
    previous pass to have released that layer's buffers.  `join(stream)`
    makes `stream` wait for everything enqueued so far."""

    def __init__(self, layers, dtype, device, fused=False):
        self.layers = layers
        self.fused = fused
        dev = torch.device(device)
        self.xd = [torch.empty((M, K), dtype=dtype, device=dev) for (_, M, K, _) in layers]
        self.yd = [torch.empty((M, N), dtype=dtype, device=dev) for (_, M, _, N) in layers]
        self.xq = [torch.empty((M, codes_width(lay.act_codes, K)), dtype=torch.uint8,
                               device=dev)
                   for (lay, M, K, _) in layers]
        self.sx = [torch.empty(M, dtype=torch.float32, device=dev) for (_, M, _, _) in layers]
        self.ws = [fused_workspace(M, K, dev) if fused else None for (_, M, K, _) in layers]
        self.s_in = torch.cuda.Stream(device=dev)
        self.s_comp = torch.cuda.Stream(device=dev)
        self.s_out = torch.cuda.Stream(device=dev)
        n = len(layers)
        self.in_done = [torch.cuda.Event() for _ in range(n)]
        self.comp_done = [torch.cuda.Event() for _ in range(n)]
        self.out_done = [torch.cuda.Event() for _ in range(n)]
        self.started = False

    def run(self, xh, yh, after=None):
        """One pass: xh[i] (host [M, K]) -> yh[i] (host [M, N]).  `after`: an
        event that every stream waits on first (for timing)."""
        for s in (self.s_in, self.s_comp, self.s_out):
            if after is not None:
                s.wait_event(after)
        for i, (lay, M, K, N) in enumerate(self.layers):
            with torch.cuda.stream(self.s_in):
                if self.started:  # the previous pass has consumed xd[i]
                    self.s_in.wait_event(self.comp_done[i])
                self.xd[i].copy_(xh[i], non_blocking=True)
                self.in_done[i].record(self.s_in)
            with torch.cuda.stream(self.s_comp):
                self.s_comp.wait_event(self.in_done[i])
                if self.started:  # the previous pass has read yd[i] back
                    self.s_comp.wait_event(self.out_done[i])
                lay(self.xd[i], fused=self.fused, workspace=self.ws[i], stream=self.s_comp,
                    Y=self.yd[i], Xq=self.xq[i], s_x=self.sx[i])
                self.comp_done[i].record(self.s_comp)
            with torch.cuda.stream(self.s_out):
                self.s_out.wait_event(self.comp_done[i])
                yh[i].copy_(self.yd[i], non_blocking=True)
                self.out_done[i].record(self.s_out)
        self.started = True

    def join(self, stream=None):
        s = torch.cuda.current_stream() if stream is None else stream
        for e in self.out_done + self.comp_done + self.in_done:
            s.wait_event(e)


def measure_peaks(stream=None, reps=5):
    """Measured peak rates on the current device (best of `reps`, CUDA events
    on `stream` around each microbenchmark launch): tcgen05 E4M3 and
    mma.sync s8 / s4 / e4m3 in TFLOP/s (2 ops per multiply-accumulate) and
    the HBM read bandwidth in GB/s; the GEMM's operand stream into shared
    memory (GB/s of shared-memory bytes, all SMs, operands L2-resident) and
    its main loop with the MMAs (TFLOP/s), for E4M3 and E2M3 operands."""
    s = torch.cuda.current_stream() if stream is None else stream
    sp = s.cuda_stream
    dev = torch.device("cuda", torch.cuda.current_device())
    buf = torch.empty(1 << 31, dtype=torch.uint8, device=dev)
    ops = ctypes.c_int64(0)

    def timed(launch):
        best = None
        for r in range(reps + 1):
            a = torch.cuda.Event(enable_timing=True)
            z = torch.cuda.Event(enable_timing=True)
            a.record(s)
            launch()
            z.record(s)
            z.synchronize()
            if r > 0:  # the first launch is a warm-up
                t = a.elapsed_time(z) * 1e-3
                best = t if best is None else min(best, t)
        return ops.value / best

    out = {}
    out["tcgen05_e4m3_tflops"] = 2e-12 * timed(lambda: _check(
        clq_peak_tcgen05_e4m3(20000, ctypes.byref(ops), sp), "clq_peak_tcgen05_e4m3"))
    for kind, name in ((0, "mma_sync_s8_tops"), (1, "mma_sync_s4_tops"),
                       (2, "mma_sync_e4m3_tflops")):
        out[name] = 2e-12 * timed(lambda: _check(
            clq_peak_mma_sync(kind, 4000, ctypes.byref(ops), sp), "clq_peak_mma_sync"))
    out["hbm_read_gbs"] = 1e-9 * timed(lambda: _check(
        clq_peak_hbm_read(buf.data_ptr(), buf.numel(), ctypes.byref(ops), sp),
        "clq_peak_hbm_read"))
    # operands of a 4096 x 1152 code array (L2-resident, like the GEMM's)
    rows, K, tiles = 4096, 1152, 48
    for codes, tag in ((CLQ_CODES_E4M3, "e4m3"), (CLQ_CODES_E2M3, "e2m3")):
        for mma in (0, 1):
            r = 1e-9 * timed(lambda: _check(
                clq_peak_operand_stream(buf.data_ptr(), rows, K, codes, mma, tiles,
                                        ctypes.byref(ops), sp), "clq_peak_operand_stream"))
            if mma:
                out["mainloop_%s_tflops" % tag] = 2e-3 * r
            else:
                out["operand_stream_%s_smem_gbs" % tag] = r
    del buf
    return {k: round(v, 1) for k, v in out.items()}
