"""GPU parity for the paper's other bit settings, W4A8 and W8A8 (Sec. 4.1):
8-bit codes (qmax 127) in the split-plane layout against the oracle's n-bit
grid, the product's accumulators bit for bit where the fp32 carrier is exact,
and whole layers against the fp64 oracle.  Tolerances: tests/parity_utils.py
(the same rules as the 4-bit path; for 8-bit codes the ratio X~ / s reaches
127, still far inside the 1e-4 tie window at fp32 resolution)."""
import numpy as np
import pytest
import torch

import oracle
from paper_2509_24416_gb300 import clq
from parity_utils import (check_codes, check_output_elementwise,
                          check_output_frobenius, check_rot, check_scales)

pytestmark = pytest.mark.gpu
DEV = torch.device("cuda:0")
TD = {"f16": torch.float16, "bf16": torch.bfloat16}
SPLIT = clq.CLQ_CODES_E4M3_SPLIT


@pytest.fixture(scope="module", autouse=True)
def _lib():
    clq.load()
    yield
    assert clq.device_status() == 0


def _decode_e4m3(byte):
    """Value of an E4M3 byte (sign, 4 exponent bits with bias 7, 3 mantissa
    bits; exponent 0 subnormal), from the format definition."""
    b = np.asarray(byte, np.int64)
    sign = np.where(b & 0x80, -1.0, 1.0)
    e = (b >> 3) & 0xF
    m = b & 0x7
    return sign * np.where(e == 0, m / 8.0 * 2.0 ** -6, (1 + m / 8.0) * 2.0 ** (e - 7.0))


def _encode_e4m3_int(v):
    """E4M3 byte of integers that the format holds exactly (|v| <= 16, or a
    multiple of 16 up to 128)."""
    v = np.asarray(v, np.int64)
    a = np.abs(v).astype(np.float64)
    f, x = np.frexp(np.where(a == 0, 1.0, a))     # a = f 2^x, f in [0.5, 1)
    e = x - 1
    m = (f * 2 - 1) * 8
    assert np.array_equal(m, np.rint(m)), "not an E4M3 value"
    byte = ((e + 7) << 3) | m.astype(np.int64)
    byte = np.where(a == 0, 0, byte) | np.where(v < 0, 0x80, 0)
    return byte.astype(np.uint8)


def _split_codes(Q, K):
    """Integer codes of a split-plane array [rows, 2K]; checks the planes."""
    Q = np.asarray(Q)
    assert Q.shape[1] == 2 * K
    hi = _decode_e4m3(Q[:, :K])
    lo = _decode_e4m3(Q[:, K:])
    assert np.all(np.mod(hi, 16) == 0) and np.abs(hi).max(initial=0) <= 128
    assert np.array_equal(lo, np.rint(lo)) and lo.min(initial=0) >= -8 and lo.max(initial=0) <= 7
    q = hi + lo
    assert np.abs(q).max(initial=0) <= 127
    return q.astype(np.int16)


def _to_split(codes):
    """int codes [rows, K] -> the split-plane layout [rows, 2K]."""
    q = np.asarray(codes, np.int64)
    h = np.floor_divide(q + 8, 16)
    return np.concatenate([_encode_e4m3_int(16 * h), _encode_e4m3_int(q - 16 * h)], axis=1)


def _inputs(M, K, dtype, seed, scale=3.0, outliers=4):
    rng = np.random.default_rng(seed)
    x = rng.standard_normal((M, K)).astype(np.float32) * scale
    if outliers:
        ch = rng.choice(K, min(outliers, K), replace=False)
        x[:, ch] *= 40
    t = torch.from_numpy(x).to(TD[dtype])
    return t, t.float().numpy()


def test_split_encoding_helpers_roundtrip():
    q = np.arange(-127, 128).reshape(1, -1)
    q = np.concatenate([q, q[:, ::-1]], axis=0)
    assert np.array_equal(_split_codes(_to_split(q), q.shape[1]), q)


@pytest.mark.parametrize("M,K,b,dtype", [(300, 1152, 64, "f16"), (129, 4608, 128, "bf16"),
                                         (77, 96, 32, "f16"), (64, 256, 1, "bf16"),
                                         (1000, 3072, 256, "f16"), (5, 16384, 16, "bf16")])
def test_rotate_quant_8bit(M, K, b, dtype):
    x_t, x32 = _inputs(M, K, dtype, seed=M + K + b)
    x32[3 % M] = 0.0
    x_t[3 % M] = 0
    perm = np.random.default_rng(K).permutation(K).astype(np.int32)
    Xq, s_x, rot = clq.rotate_quant_act(x_t.to(DEV), torch.from_numpy(perm).to(DEV), b,
                                        codes=SPLIT, with_rot=True)
    torch.cuda.synchronize()
    assert Xq.shape == (M, 2 * K)
    _, os_, orot, oc = oracle.rotate_quant_act(x32, perm, b, bits=8)
    check_rot(rot.cpu().numpy(), orot)
    check_scales(s_x.cpu().numpy(), os_)
    check_codes(_split_codes(Xq.cpu().numpy(), K), oc, orot, os_)
    assert s_x[3 % M].item() == 0.0


def test_prepare_weights_8bit_with_and_without_clip():
    N, K, b = 257, 1152, 64
    rng = np.random.default_rng(9)
    w_t = torch.from_numpy((rng.standard_normal((N, K)) * 0.05).astype(np.float32)).to(torch.bfloat16)
    w32 = w_t.float().numpy()
    perm = rng.permutation(K).astype(np.int32)
    permd = torch.from_numpy(perm).to(DEV)
    _, _, orot0, _ = oracle.prepare_weights(w32, perm, b, bits=8)
    clip = (np.max(np.abs(orot0), axis=1) * 0.6).astype(np.float32)
    for c in (None, clip):
        Wq, s_w, rot = clq.prepare_weights(w_t.to(DEV), permd, b,
                                           None if c is None else torch.from_numpy(c).to(DEV),
                                           with_rot=True, codes=SPLIT)
        torch.cuda.synchronize()
        _, os_, orot, oc = oracle.prepare_weights(w32, perm, b, c, bits=8)
        check_rot(rot.cpu().numpy(), orot)
        check_scales(s_w.cpu().numpy(), os_)
        gq = _split_codes(Wq.cpu().numpy(), K)
        check_codes(gq, oc, orot, os_)
        if c is not None:
            assert np.abs(gq).max() == 127 and np.count_nonzero(np.abs(gq) == 127) > N


def _product_case(qx, qw, s_x, s_w, b, w_bits, dtype, bias=None):
    """GPU product fed the given codes (activations split, weights split or
    E4M3) against the oracle's exact accumulators and fp64 epilogue."""
    M, K = qx.shape
    Xq = torch.from_numpy(_to_split(qx)).to(DEV)
    Wc = _to_split(qw) if w_bits == 8 else _encode_e4m3_int(qw)
    W = torch.from_numpy(Wc).to(DEV)
    bias_t = None if bias is None else torch.from_numpy(bias).to(TD[dtype]).to(DEV)
    b32 = None if bias_t is None else bias_t.float().cpu().numpy()
    Y, gacc = clq.linear(Xq, torch.from_numpy(s_x).to(DEV), W, torch.from_numpy(s_w).to(DEV),
                         b, K, bias_t, out_dtype=TD[dtype], with_acc=True)
    torch.cuda.synchronize()
    y64, acc = oracle.quant_linear(qx, s_x, qw, s_w, b, b32)
    return Y.float().cpu().numpy(), gacc.cpu().numpy(), y64, acc, b32


@pytest.mark.parametrize("w_bits", [4, 8])
@pytest.mark.parametrize("M,N,K", [(1, 1, 32), (17, 64, 128), (300, 600, 1152),
                                   (129, 257, 96), (256, 512, 4608), (130, 200, 16384)])
def test_linear_8bit_acc_exact_and_output(w_bits, M, N, K):
    rng = np.random.default_rng(M * 7 + N + K + w_bits)
    qx = rng.integers(-127, 128, (M, K)).astype(np.int16)
    qw = rng.integers(-127 if w_bits == 8 else -7, 128 if w_bits == 8 else 8, (N, K)).astype(np.int16)
    s_x = rng.uniform(0.01, 0.1, M).astype(np.float32)
    s_w = rng.uniform(0.001, 0.01, N).astype(np.float32)
    bias = (rng.standard_normal(N) * 0.1).astype(np.float32)
    for dtype in ("f16", "bf16"):
        y, gacc, y64, acc, b32 = _product_case(qx, qw, s_x, s_w, 32, w_bits, dtype, bias)
        # random codes keep every partial sum far below 2^24: exact at any K
        assert np.array_equal(gacc, acc)
        check_output_elementwise(y, y64, acc, s_x, s_w, 32, b32, dtype)
        check_output_frobenius(y, y64)


@pytest.mark.parametrize("K", [4608, 16384])
def test_w4a8_carrier_exact_at_extremes(K):
    """Every code at its extreme: |acc| reaches 127 * 7 * K (14.6e6 at
    K = 16384, just below 2^24), and mixed rows rise to half of that and
    return to 0.  The W4A8 accumulators must stay exact."""
    M, N = 136, 264
    rng = np.random.default_rng(K)
    qx = np.where(rng.random((M, K)) < 0.5, -127, 127).astype(np.int16)
    qw = np.where(rng.random((N, K)) < 0.5, -7, 7).astype(np.int16)
    qx[:8] = 127
    qw[:8] = 7
    qw[8:16] = -7
    qx[8:16, : K // 2] = 127
    qx[8:16, K // 2:] = -127
    ones_x = np.ones(M, np.float32)
    ones_w = np.ones(N, np.float32)
    _, gacc, _, acc, _ = _product_case(qx, qw, ones_x, ones_w, 32, 4, "bf16")
    assert np.array_equal(gacc, acc)
    assert acc[0, 0] == 889 * K


@pytest.mark.parametrize("K", [896, 4096, 16384])
def test_w8a8_carrier_exact_at_extremes(K):
    """W8A8 with every code at +-127: |acc| reaches 16129 K (2.6e8 at
    K = 16384), far past 2^24, and mixed rows rise to half of that and return
    to 0.  The plane products are accumulated apart (multiples of 256, of 16
    and plain integers) and added as integers, so the accumulators stay exact
    at every K."""
    M, N = 130, 140
    rng = np.random.default_rng(K)
    qx = np.where(rng.random((M, K)) < 0.5, -127, 127).astype(np.int16)
    qw = np.where(rng.random((N, K)) < 0.5, -127, 127).astype(np.int16)
    qx[:8] = 127
    qw[:8] = 127
    qw[8:16] = -127
    qx[8:16, : K // 2] = 127
    qx[8:16, K // 2:] = -127
    qx[16:24] = rng.integers(-127, 128, (8, K))   # every code value
    ones_x = np.ones(M, np.float32)
    ones_w = np.ones(N, np.float32)
    y, gacc, y64, acc, _ = _product_case(qx, qw, ones_x, ones_w, 32, 8, "bf16")
    assert np.array_equal(gacc, acc)
    assert acc[0, 0] == 16129 * K
    check_output_elementwise(y, y64, acc, ones_x, ones_w, 32, None, "bf16")


@pytest.mark.parametrize("a_bits,w_bits", [(8, 4), (8, 8)])
@pytest.mark.parametrize("dtype", ["f16", "bf16"])
def test_layer_8bit_end_to_end(a_bits, w_bits, dtype):
    """X -> rotate-quant (8-bit split) -> product with weights prepared at
    w_bits, against the oracle layer at the same bit setting."""
    M, N, K, b = 384, 768, 1152, 64
    x_t, x32 = _inputs(M, K, dtype, seed=a_bits + w_bits)
    rng = np.random.default_rng(3)
    w_t = torch.from_numpy((rng.standard_normal((N, K)) * 0.02).astype(np.float32)).to(TD[dtype])
    bias_t = torch.from_numpy((rng.standard_normal(N) * 0.01).astype(np.float32)).to(TD[dtype])
    scores = clq.outlier_scores(x_t.to(DEV)[None])
    perm = clq.build_permutation(scores)
    permd = perm.to(DEV)
    w_layout = SPLIT if w_bits == 8 else clq.CLQ_CODES_E4M3
    Wq, s_w = clq.prepare_weights(w_t.to(DEV), permd, b, codes=w_layout)
    Xq, s_x = clq.rotate_quant_act(x_t.to(DEV), permd, b, codes=SPLIT)
    Y = clq.linear(Xq, s_x, Wq, s_w, b, K, bias_t.to(DEV), out_dtype=TD[dtype])
    torch.cuda.synchronize()
    p = perm.numpy()
    _, os_w, orot_w, owc = oracle.prepare_weights(w_t.float().numpy(), p, b, bits=w_bits)
    _, os_x, orot, oxc = oracle.rotate_quant_act(x32, p, b, bits=a_bits)
    gw = (_split_codes(Wq.cpu().numpy(), K) if w_bits == 8
          else _decode_e4m3(Wq.cpu().numpy()).astype(np.int16))
    check_codes(gw, owc, orot_w, os_w)
    gx = _split_codes(Xq.cpu().numpy(), K)
    check_codes(gx, oxc, orot, os_x)
    b32 = bias_t.float().numpy()
    y = Y.float().cpu().numpy()
    y64 = oracle.obs_linear(x32, p, b, owc, os_w, b32, a_bits=a_bits)
    check_output_frobenius(y, y64)
    # with the GPU's own codes and scales the product is exact up to output rounding
    y64g, accg = oracle.quant_linear(gx, s_x.cpu().numpy(), gw, s_w.cpu().numpy(), b, b32)
    check_output_elementwise(y, y64g, accg, s_x.cpu().numpy(), s_w.cpu().numpy(), b, b32, dtype)
    # more bits, less error than W4A4 on the same layer
    ref = oracle.linear_fp64(x32, w_t.float().numpy(), b32)
    oWq4, os_w4, _, _ = oracle.prepare_weights(w_t.float().numpy(), p, b)
    y4 = oracle.fused_linear(x32, p, b, oWq4, os_w4, b32)
    assert np.linalg.norm(y - ref) < np.linalg.norm(y4 - ref)


@pytest.mark.parametrize("a_bits,w_bits", [(4, 4), (8, 4), (8, 8)])
def test_prepared_linear_bit_settings(a_bits, w_bits):
    """The layer object at each bit setting equals the explicit calls, and
    survives a state-dict round trip."""
    M, N, K, b = 200, 300, 1152, 64
    x_t, _ = _inputs(M, K, "bf16", seed=11)
    rng = np.random.default_rng(12)
    W = torch.from_numpy((rng.standard_normal((N, K)) * 0.02).astype(np.float32)).to(torch.bfloat16)
    perm = torch.from_numpy(rng.permutation(K).astype(np.int32)).to(DEV)
    X = x_t.to(DEV)
    layer = clq.PreparedLinear.from_weight(W.to(DEV), perm, b, a_bits=a_bits, w_bits=w_bits)
    assert layer.w_bits == w_bits and layer.a_bits == a_bits
    Y = layer(X)
    codes = layer.act_codes   # split planes at A8, else the weights' 4-bit layout
    Xq, s_x = clq.rotate_quant_act(X, perm, b, codes=codes)
    Y2 = clq.linear(Xq, s_x, layer.We, layer.s_w, b, K, out_dtype=X.dtype)
    again = clq.PreparedLinear.from_state_dict(layer.state_dict())(X)
    torch.cuda.synchronize()
    assert torch.equal(Y, Y2) and torch.equal(Y, again)
    if a_bits == 4:
        assert torch.equal(layer(X, fused=True), Y)
    else:
        with pytest.raises(ValueError):
            layer(X, fused=True)


@pytest.mark.parametrize("li", [0, 3])
@pytest.mark.parametrize("a_bits,w_bits", [(8, 4), (8, 8)])
def test_pixart_layer_full_size_sampled_rows_8bit(li, a_bits, w_bits):
    """The PixArt-1024 layer at its full 8192 tokens, every row through the
    GPU as the bench launches it, 42 sampled rows against the oracle."""
    from paper_2509_24416_gb300 import synth
    cfg = synth.WORKLOADS["pixart_1024"]
    d = synth.layer_inputs(cfg, li)
    b, K = d["b"], d["K"]
    M = cfg["M"]
    rows = np.sort(np.concatenate([np.random.default_rng(li).choice(M, 40, replace=False),
                                   [0, M - 1]]))
    perm = oracle.build_permutation(oracle.outlier_scores(d["calib"]))
    permd = torch.from_numpy(perm).to(DEV)
    layout_w = SPLIT if w_bits == 8 else clq.CLQ_CODES_E4M3
    Wq, s_w = clq.prepare_weights(d["W"].to(DEV), permd, b, codes=layout_w)
    Xq, s_x, rot = clq.rotate_quant_act(d["X"].to(DEV), permd, b, codes=SPLIT, with_rot=True)
    Y = clq.linear(Xq, s_x, Wq, s_w, b, K, d["bias"].to(DEV), out_dtype=TD[d["dtype"]])
    torch.cuda.synchronize()
    _, os_w, orot_w, owc = oracle.prepare_weights(d["W32"], perm, b, bits=w_bits)
    _, os_x, orot, oxc = oracle.rotate_quant_act(d["X32"][rows], perm, b, bits=8)
    check_rot(rot.cpu().numpy()[rows], orot)
    check_scales(s_x.cpu().numpy()[rows], os_x)
    check_codes(_split_codes(Xq.cpu().numpy()[rows], K), oxc, orot, os_x)
    gw = (_split_codes(Wq.cpu().numpy(), K) if w_bits == 8
          else _decode_e4m3(Wq.cpu().numpy()).astype(np.int16))
    check_codes(gw, owc, orot_w, os_w)
    y64, _ = oracle.quant_linear(oxc, os_x, owc, os_w, b, d["bias32"])
    check_output_frobenius(Y.float().cpu().numpy()[rows], y64)
