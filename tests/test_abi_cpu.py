"""CPU-only checks of the C ABI: the library loads, exports every symbol that
include/clq.h declares, rejects bad arguments on the host before any launch,
and its host column-swap builder matches the oracle's."""
import ctypes
import os
import re

import numpy as np
import pytest
import torch

import oracle
from paper_2509_24416_gb300 import build, clq

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    build.build()
    return clq.load()


def declared_functions():
    text = open(os.path.join(ROOT, "include", "clq.h")).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(clq_[a-z0-9_]+)\s*\(", text)))


def test_header_matches_binding():
    assert declared_functions() == sorted(clq.EXPORTS)


def test_all_symbols_exported(lib):
    for name in declared_functions():
        assert hasattr(lib, name), name


def test_status_strings(lib):
    for code, name in clq.STATUS.items():
        assert lib.clq_status_string(code).decode().startswith(name)
    assert lib.clq_version() == 102


P = 1 << 20  # a fake, 16-byte aligned "device" address; never dereferenced


@pytest.mark.parametrize("args,code", [
    # (X, dtype, M, K, ldx, perm, b, codes, Xq, s_x, rot) -> expected status
    ((P, 2, 4, 64, 64, P, 32, 0, P, P, None), 1),      # bad dtype
    ((P, 0, 4, 64, 64, P, 32, 4, P, P, None), 1),      # bad code layout
    ((P, 0, 4, 64, 64, P, 32, 3, P, P, None), 2),      # E2M3 needs K % 128
    ((P, 0, 4, 128, 128, P, 32, 3, P + 16, P, None), 3),  # E2M3 array 32-byte aligned
    ((P, 0, -1, 64, 64, P, 32, 0, P, P, None), 1),     # negative M
    ((P, 0, 4, 64, 64, P, 3, 0, P, P, None), 2),       # b not a power of two
    ((P, 0, 4, 64, 64, P, 512, 1, P, P, None), 2),     # b > 256
    ((P, 0, 4, 48, 48, P, 16, 0, P, P, None), 2),      # K % 32
    ((P, 0, 4, 1152, 1152, P, 256, 0, P, P, None), 2), # K % b (1152 / 256)
    ((P, 0, 4, 32768, 32768, P, 32, 0, P, P, None), 2),  # K too large
    ((P, 0, 4, 64, 32, P, 32, 0, P, P, None), 2),      # ldx < K
    ((P, 0, 4, 64, 68, P, 32, 0, P, P, None), 3),      # ldx % 8
    ((None, 0, 4, 64, 64, P, 32, 0, P, P, None), 1),   # null X
    ((P, 0, 4, 64, 64, None, 32, 1, P, P, None), 1),   # null perm
    ((P + 8, 0, 4, 64, 64, P, 32, 0, P, P, None), 3),  # misaligned X
    ((P, 0, 4, 64, 64, P, 32, 1, P + 4, P, None), 3),  # misaligned Xq
    ((P, 0, 0, 64, 64, None, 32, 0, None, None, None), 0),  # empty: no-op
])
def test_rotate_quant_host_validation(lib, args, code):
    assert clq.clq_rotate_quant_act(*args, None) == code


@pytest.mark.parametrize("args,code", [
    # (Xq, x_codes, s_x, W, w_codes, s_w, bias, M, N, K, b, out_dtype, Y, acc)
    ((P, 0, P, P, 0, P, None, 4, 4, 64, 32, 3, P, None), 1),     # bad out dtype
    ((P, 0, P, P, 2, P, None, 4, 4, 64, 32, 0, P, None), 1),     # bad w layout
    ((P, 5, P, P, 0, P, None, 4, 4, 64, 32, 0, P, None), 1),     # bad x layout
    ((P, 0, P, P, 0, P, None, 4, -2, 64, 32, 0, P, None), 1),    # negative N
    ((P, 1, P, P, 1, P, None, 4, 4, 96, 64, 0, P, None), 2),     # K % b
    ((P, 0, P, P, 0, P, None, 4, 4, 64, 32, 0, P + 2, None), 3), # misaligned Y
    ((P, 0, P, P, 0, P, P + 1, 4, 4, 64, 32, 0, P, None), 3),    # misaligned bias
    ((None, 0, P, P, 0, P, None, 4, 4, 64, 32, 0, P, None), 1),  # null Xq
    ((None, 0, None, None, 0, None, None, 0, 4, 64, 32, 0, None, None), 0),
    ((None, 1, None, None, 1, None, None, 4, 0, 64, 32, 0, None, None), 0),
])
def test_w4a4_host_validation(lib, args, code):
    assert clq.clq_w4a4_linear(*args, None) == code


@pytest.mark.parametrize("args,code", [
    # (Xq, x_codes, s_x, W, w_codes, s_w, bias, M, N, K, b, out_dtype, Y, acc)
    ((P, 2, P, P, 0, P, None, 4, 4, 64, 32, 0, P, None), 4),     # W4A8, packed W
    ((P, 0, P, P, 2, P, None, 4, 4, 64, 32, 0, P, None), 4),     # W8A4
    ((P, 1, P, P, 2, P, None, 4, 4, 64, 32, 0, P, None), 4),     # W8A4
    ((P, 5, P, P, 1, P, None, 4, 4, 64, 32, 0, P, None), 1),     # bad x layout
    ((P, 3, P, P, 1, P, None, 4, 4, 128, 32, 0, P, None), 4),    # E2M3 with E4M3
    ((P, 1, P, P, 3, P, None, 4, 4, 128, 32, 0, P, None), 4),    # E4M3 with E2M3
    ((P, 3, P, P, 3, P, None, 4, 4, 64, 32, 0, P, None), 2),     # E2M3, K % 128
    ((P, 3, P, P + 16, 3, P, None, 4, 4, 128, 32, 0, P, None), 3),  # E2M3 W alignment
    ((None, 3, None, None, 3, None, None, 0, 4, 128, 32, 0, None, None), 0),
    ((P, 2, P, P, 2, P, None, 4, 4, 48, 16, 0, P, None), 2),     # K % 32
    ((P, 2, P, P, 1, P, None, 4, 4, 64, 32, 0, P + 2, None), 3), # misaligned Y
    ((None, 2, None, None, 2, None, None, 0, 4, 64, 32, 0, None, None), 0),
])
def test_linear_host_validation(lib, args, code):
    assert clq.clq_linear(*args, None) == code


def test_prepare_weights_codes_host_validation(lib):
    # (W, dtype, N, K, ldw, perm, b, clip, w_codes, Wq, s_w, rot, stream)
    assert clq.clq_prepare_weights_codes(P, 0, 4, 64, 64, P, 32, None, 4, P, P,
                                         None, None) == 1
    assert clq.clq_prepare_weights_codes(P, 0, 4, 64, 64, P, 32, None, 3, P, P,
                                         None, None) == 2          # E2M3, K % 128
    assert clq.clq_prepare_weights_codes(P, 0, 4, 64, 64, P, 32, P + 2, 2, P,
                                         P, None, None) == 3
    assert clq.clq_prepare_weights_codes(P, 0, 4, 64, 64, P, 5, None, 2, P, P,
                                         None, None) == 2
    assert clq.clq_prepare_weights_codes(None, 0, 0, 64, 64, None, 32, None, 2,
                                         None, None, None, None) == 0


def test_asym_host_validation(lib):
    # rotate-quant asym: (X, dtype, M, K, ldx, perm, b, codes, Xq, delta, lo, rot, stream)
    assert clq.clq_rotate_quant_act_asym(P, 0, 4, 64, 64, P, 32, 1, P, P, None, None,
                                         None) == 1                    # lo missing
    assert clq.clq_rotate_quant_act_asym(P, 0, 4, 64, 64, P, 32, 5, P, P, P, None,
                                         None) == 1                    # bad layout
    assert clq.clq_rotate_quant_act_asym(P, 0, 4, 128, 128, P, 32, 3, P, P, P, None,
                                         None) == 4                    # E2M3: no -8
    assert clq.clq_rotate_quant_act_asym(P, 0, 4, 64, 64, P, 32, 1, P, P, P + 2, None,
                                         None) == 3                    # misaligned lo
    assert clq.clq_rotate_quant_act_asym(None, 0, 0, 64, 64, None, 32, 1, None, None,
                                         None, None, None) == 0        # empty
    # code sums: (W, codes, N, K, wsum, stream)
    assert clq.clq_weight_code_sums(P, 5, 4, 64, P, None) == 1
    assert clq.clq_weight_code_sums(P, 3, 4, 64, P, None) == 2     # E2M3, K % 128
    assert clq.clq_weight_code_sums(P, 1, 4, 48, P, None) == 2
    assert clq.clq_weight_code_sums(P, 1, 4, 64, P + 1, None) == 3
    assert clq.clq_weight_code_sums(None, 1, 0, 64, None, None) == 0
    # linear asym: (Xq, xc, delta, lo, W, wc, s_w, wsum, bias, M, N, K, b, dt, Y, acc, st)
    assert clq.clq_linear_asym(P, 0, P, P, P, 1, P, P, None, 4, 4, 64, 32, 0, P, None,
                               None) == 4                              # packed A
    assert clq.clq_linear_asym(P, 1, P, P, P, 2, P, P, None, 4, 4, 64, 32, 0, P, None,
                               None) == 4                              # W8A4
    assert clq.clq_linear_asym(P, 1, P, None, P, 1, P, P, None, 4, 4, 64, 32, 0, P, None,
                               None) == 1                              # lo missing
    assert clq.clq_linear_asym(P, 1, P, P, P, 1, P, P + 2, None, 4, 4, 64, 32, 0, P, None,
                               None) == 3                              # misaligned wsum
    assert clq.clq_linear_asym(P, 5, P, P, P, 1, P, P, None, 4, 4, 64, 32, 0, P, None,
                               None) == 1                              # bad layout


def test_clip_search_host_validation(lib):
    import ctypes
    grid = (ctypes.c_float * 3)(0.0, 0.005, 0.01)
    bad = (ctypes.c_float * 2)(0.0, 1.5)
    g = ctypes.addressof(grid)
    assert clq.clq_clip_search_workspace_size(256, 128, 1152, g, 3) > 0
    assert clq.clq_clip_search_workspace_size(256, 128, 1152, ctypes.addressof(bad), 2) == 0
    assert clq.clq_clip_search_workspace_size(256, 128, 48, g, 3) == 0
    assert clq.clq_clip_search_workspace_size(0, 128, 1152, g, 3) == 0
    errs = (ctypes.c_double * 3)()
    best = ctypes.c_int32(0)
    e, bp = ctypes.addressof(errs), ctypes.addressof(best)
    # (W, dtype, N, K, ldw, perm, b, X, M, ldx, Yref, bias, grid, G, clip,
    #  errors, best, ws, ws_bytes, stream)
    assert clq.clq_clip_search(P, 0, 8, 64, 64, P, 32, P, 8, 64, P, None, g, 3, P, e, bp,
                               P, 16, None) == 1                       # workspace small
    assert clq.clq_clip_search(P, 0, 8, 64, 64, P, 3, P, 8, 64, P, None, g, 3, P, e, bp,
                               P, 1 << 30, None) == 2                  # b
    assert clq.clq_clip_search(P, 0, 8, 64, 64, P, 32, P, 8, 64, P, None,
                               ctypes.addressof(bad), 2, P, e, bp, P, 1 << 30, None) == 1
    assert clq.clq_clip_search(P, 0, 8, 64, 64, P, 32, P, 8, 64, P, None, g, 3, P, e, bp,
                               P + 16, 1 << 30, None) == 3              # ws alignment
    assert clq.clq_clip_search(P, 0, 0, 64, 64, P, 32, P, 8, 64, P, None, g, 3, P, e, bp,
                               P, 1 << 30, None) == 1                  # N = 0


def test_fused_and_prepare_host_validation(lib):
    ws = clq.clq_fused_linear_workspace_size(256, 1152)
    # 256 x 1152 E4M3 codes, 256 scales, 2 block counters + 1 tile counter
    assert ws == 294912 + 1024 + 256
    assert clq.clq_fused_linear_workspace_size(4, 48) == 0
    # (X, dtype, M, K, ldx, perm, b, W, w_format, s_w, bias, N, Y, ws, bytes)
    assert clq.clq_fused_linear(P, 0, 4, 64, 64, P, 7, P, 0, P, None, 4, P, P,
                                1 << 20, None) == 2
    assert clq.clq_fused_linear(P, 0, 4, 64, 64, P, 32, P, 0, P, None, 0, P,
                                P, 1 << 20, None) == 0
    assert clq.clq_fused_linear(P, 0, 4, 64, 64, P, 32, P, 0, P, None, 4, P,
                                P, 16, None) == 1         # workspace too small
    assert clq.clq_fused_linear(P, 0, 4, 64, 64, P, 32, P, 0, P, None, 4, P,
                                P + 16, 1 << 20, None) == 3  # 256-B alignment
    assert clq.clq_fused_linear(P, 0, 4, 64, 64, P, 32, P, 5, P, None, 4, P,
                                P, 1 << 20, None) == 1    # bad w_format
    assert clq.clq_fused_linear(P, 0, 4, 64, 64, P, 32, P, 3, P, None, 4, P,
                                P, 1 << 20, None) == 2    # E2M3 weights, K % 128
    assert clq.clq_fused_linear(P, 0, 4, 128, 128, P, 32, P + 16, 3, P, None, 4, P,
                                P, 1 << 20, None) == 3    # E2M3 weights, alignment
    # convert: (src, src_codes, dst, dst_codes, rows, K, stream)
    assert clq.clq_convert_codes(P, 0, P, 5, 4, 128, None) == 1
    assert clq.clq_convert_codes(P, 0, P, 3, 4, 64, None) == 2     # E2M3, K % 128
    assert clq.clq_convert_codes(P, 0, P, 1, 4, 48, None) == 2     # K % 32
    assert clq.clq_convert_codes(P, 0, P + 16, 3, 4, 128, None) == 3
    assert clq.clq_convert_codes(P + 8, 0, P, 1, 4, 128, None) == 3
    assert clq.clq_convert_codes(None, 0, None, 3, 0, 128, None) == 0
    assert clq.clq_convert_codes(None, 0, P, 3, 4, 128, None) == 1
    assert clq.clq_prepare_weights(P, 0, 4, 64, 64, P, 32, P + 2, P, P, None,
                                   None) == 3
    assert clq.clq_expand_weights(P, 4, 48, P, None) == 2
    assert clq.clq_expand_weights(P, 0, 64, None, None) == 0
    assert clq.clq_expand_weights(P + 8, 4, 64, P, None) == 3
    assert clq.clq_outlier_scores(P, 0, 0, 4, 4, P, None) == 1
    assert clq.clq_selftest_bounded_wait(10, None) == 1
    assert clq.clq_get_device_status(None, None) == 1


def test_outlier_metric_host_validation(lib):
    assert clq.clq_outlier_scores_metric(P, 0, 2, 8, 4, 5, P, None) == 1      # metric
    assert clq.clq_outlier_scores_metric(P, 0, 2, 8, 4, -1, P, None) == 1
    assert clq.clq_outlier_scores_metric(P, 0, 2, 16385, 4, 1, P, None) == 2  # T limit
    assert clq.clq_outlier_scores_metric(P, 2, 2, 8, 4, 1, P, None) == 1      # dtype
    assert clq.clq_outlier_scores_metric(None, 0, 2, 8, 4, 1, P, None) == 1
    assert clq.clq_outlier_scores_metric(P + 1, 0, 2, 8, 4, 1, P, None) == 3  # alignment
    assert clq.clq_outlier_scores_metric(P, 0, 0, 8, 4, 1, P, None) == 1      # B < 1


def test_peak_microbenchmark_host_validation(lib):
    ops = ctypes.c_int64(0)
    assert clq.clq_peak_tcgen05_e4m3(0, ctypes.byref(ops), None) == 1      # iters < 1
    assert clq.clq_peak_tcgen05_e4m3(10, None, None) == 1                  # null ops
    assert clq.clq_peak_mma_sync(3, 10, ctypes.byref(ops), None) == 1      # bad kind
    assert clq.clq_peak_mma_sync(0, 2000000, ctypes.byref(ops), None) == 1  # iters > 1e6
    assert clq.clq_peak_hbm_read(P, 100, ctypes.byref(ops), None) == 1     # bytes % 16
    assert clq.clq_peak_hbm_read(P + 4, 64, ctypes.byref(ops), None) == 3  # alignment
    assert clq.clq_peak_hbm_read(None, 64, ctypes.byref(ops), None) == 1
    E4, E2, PK = clq.CLQ_CODES_E4M3, clq.CLQ_CODES_E2M3, clq.CLQ_CODES_INT4_PACKED
    ok = (P, 256, 128, E4, 0, 1, ctypes.byref(ops), None)
    for i, bad, want in ((3, PK, 1), (4, 2, 1), (4, -1, 1), (5, 0, 1), (5, 100001, 1),
                         (1, 255, 2), (1, 384, 2), (2, 64, 2), (2, 192, 2), (2, 16512, 2),
                         (0, P + 16, 3), (0, None, 1)):
        args = list(ok)
        args[i] = bad
        assert clq.clq_peak_operand_stream(*args) == want, (i, bad)
    assert clq.clq_peak_operand_stream(P, 256, 128, E2, 2, 1, ctypes.byref(ops), None) == 1
    assert clq.clq_peak_operand_stream(P, 256, 128, E4, 0, 1, None, None) == 1
    # rotate-quant memory floor: X, M, K, Q, S, ops
    ok = (P, 8, 1152, P, P, ctypes.byref(ops), None)
    for i, bad, want in ((0, None, 1), (3, None, 1), (4, None, 1), (5, None, 1),
                         (1, 0, 2), (2, 32, 2), (2, 1120, 2), (2, 16448, 2),
                         (0, P + 8, 3), (3, P + 4, 3), (4, P + 2, 3)):
        args = list(ok)
        args[i] = bad
        assert clq.clq_peak_rq_stream(*args) == want, (i, bad)


@pytest.mark.parametrize("K,seed", [(1, 0), (2, 1), (7, 2), (64, 3),
                                    (1152, 4), (4608, 5)])
def test_build_permutation_matches_oracle(lib, K, seed):
    rng = np.random.default_rng(seed)
    scores = rng.uniform(0, 1, K).astype(np.float32)
    scores[rng.choice(K, max(1, K // 100), replace=False)] *= 40
    scores[: K // 3] = np.round(scores[: K // 3] * 4) / 4  # many exact ties
    got = clq.build_permutation(torch.from_numpy(scores)).numpy()
    assert np.array_equal(got, oracle.build_permutation(scores))


def test_build_permutation_rejects_nan(lib):
    s = torch.tensor([1.0, float("nan"), 2.0])
    perm = torch.empty(3, dtype=torch.int32)
    assert clq.clq_build_permutation(s.data_ptr(), 3, perm.data_ptr()) == 1


def test_missing_library_fails_loudly(monkeypatch, tmp_path):
    monkeypatch.setattr(clq, "_lib", None)
    monkeypatch.setattr(clq, "LIB_PATH", str(tmp_path / "nope.so"))
    with pytest.raises(RuntimeError, match="not built"):
        clq.load()


def test_binding_rejects_mis_sized_output_buffers():
    """The C ABI cannot check buffer sizes; the binding checks what it is
    handed against what the call will write, before any launch."""
    import torch
    X = torch.zeros((4, 64), dtype=torch.float16)
    perm = torch.arange(64, dtype=torch.int32)
    small = torch.empty((4, 64), dtype=torch.uint8)      # split layout needs [4, 128]
    with pytest.raises(ValueError):
        clq.rotate_quant_act(X, perm, 32, clq.CLQ_CODES_E4M3_SPLIT, Xq=small)
    with pytest.raises(ValueError):
        clq.rotate_quant_act(X, perm, 32, clq.CLQ_CODES_E4M3,
                             s_x=torch.empty(3, dtype=torch.float32))
    with pytest.raises(ValueError):
        clq.rotate_quant_act_asym(X, perm, 32, clq.CLQ_CODES_E4M3,
                                  lo=torch.empty(4, dtype=torch.float64))
    Xq = torch.empty((4, 64), dtype=torch.uint8)
    W = torch.empty((8, 64), dtype=torch.uint8)
    s = torch.empty(8, dtype=torch.float32)
    with pytest.raises(ValueError):
        clq.linear(Xq, s[:4], W, s, 32, 64, Y=torch.empty((4, 7), dtype=torch.float16))
