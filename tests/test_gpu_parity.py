"""GPU parity: the CUDA path through the C ABI against the CPU oracle, element
by element on the same seeded inputs.  Tolerances: tests/parity_utils.py."""
import numpy as np
import pytest
import torch

import oracle
from paper_2509_24416_gb300 import clq, synth
from parity_utils import (check_codes, check_output_elementwise,
                          check_output_frobenius, check_rot, check_scales)

pytestmark = pytest.mark.gpu
DEV = torch.device("cuda:0")
TD = {"f16": torch.float16, "bf16": torch.bfloat16}


@pytest.fixture(scope="module", autouse=True)
def _lib():
    clq.load()
    yield
    assert clq.device_status() == 0


def _inputs(M, K, dtype, seed, scale=3.0, outliers=4):
    rng = np.random.default_rng(seed)
    x = rng.standard_normal((M, K)).astype(np.float32) * scale
    if outliers:
        ch = rng.choice(K, min(outliers, K), replace=False)
        x[:, ch] *= 40
    t = torch.from_numpy(x).to(TD[dtype])
    return t, t.float().numpy()


def _perm(K, kind, seed=0):
    if kind == "identity":
        return np.arange(K, dtype=np.int32)
    if kind == "reversed":
        return np.arange(K - 1, -1, -1, dtype=np.int32)
    return np.random.default_rng(seed).permutation(K).astype(np.int32)


def _decode_e4m3(byte):
    """Value of an E4M3 byte (1 sign, 4 exponent bits with bias 7, 3 mantissa
    bits; exponent 0 is subnormal), written out from the format definition."""
    b = np.asarray(byte, np.int64)
    sign = np.where(b & 0x80, -1.0, 1.0)
    e = (b >> 3) & 0xF
    m = b & 0x7
    val = np.where(e == 0, m / 8.0 * 2.0 ** -6, (1 + m / 8.0) * 2.0 ** (e - 7.0))
    return sign * val


def _decode_e2m3(field):
    """Value of a 6-bit E2M3 field (1 sign bit, 2 exponent bits with bias 1,
    3 mantissa bits; exponent 0 is subnormal), from the format definition."""
    f = np.asarray(field, np.int64)
    sign = np.where(f & 0x20, -1.0, 1.0)
    e = (f >> 3) & 0x3
    m = f & 0x7
    val = np.where(e == 0, m / 8.0, (1 + m / 8.0) * 2.0 ** (e - 1.0))
    return sign * val


def _e2m3_fields(Q, K):
    """6-bit fields of an E2M3 code array [rows, 3K/4]: each 12-byte group is
    one little-endian 96-bit field holding 16 codes, code i in bits 6i.."""
    Q = np.ascontiguousarray(Q, np.uint8)
    rows = Q.shape[0]
    bits = np.unpackbits(Q.reshape(rows, K // 16, 12), axis=-1, bitorder="little")
    bits = bits.reshape(rows, K // 16, 16, 6).astype(np.int64)
    return (bits << np.arange(6)).sum(-1).reshape(rows, K)


def _encode_e2m3(codes):
    """Host encoder of integer codes in [-7, 7] into the E2M3 layout, from the
    format definition: |q| = (1 + m / 8) 2^(e - 1), e >= 1 (0 for q = 0)."""
    codes = np.asarray(codes, np.int64)
    rows, K = codes.shape
    mag = np.abs(codes)
    e = np.where(mag == 0, 0, np.floor(np.log2(np.maximum(mag, 1))).astype(np.int64) + 1)
    m = np.where(mag == 0, 0, (mag * 8 // (1 << np.maximum(e - 1, 0))) - 8)
    f = (np.where(codes < 0, 0x20, 0) | (e << 3) | m).astype(np.int64)
    assert np.array_equal(_decode_e2m3(f), codes.astype(np.float64))
    bits = ((f.reshape(rows, K // 16, 16, 1) >> np.arange(6)) & 1).astype(np.uint8)
    return np.packbits(bits.reshape(rows, K // 16, 96), axis=-1,
                       bitorder="little").reshape(rows, K // 4 * 3)


def _codes(Xq, K):
    """Integer codes of a GPU code array in any 4-bit layout."""
    Xq = np.asarray(Xq)
    if 4 * Xq.shape[1] == 3 * K:
        v = _decode_e2m3(_e2m3_fields(Xq, K))
        assert np.array_equal(v, np.rint(v)) and np.abs(v).max(initial=0) <= 7
        return v.astype(np.int8)
    if Xq.shape[1] == K:
        v = _decode_e4m3(Xq)
        assert np.array_equal(v, np.rint(v)) and np.abs(v).max(initial=0) <= 7
        return v.astype(np.int8)
    return oracle.unpack_int4(Xq)


def _rq_gpu(x, perm, b, codes=clq.CLQ_CODES_INT4_PACKED):
    Xq, s_x, rot = clq.rotate_quant_act(x.to(DEV), torch.from_numpy(perm).to(DEV),
                                        b, codes, with_rot=True)
    torch.cuda.synchronize()
    return Xq.cpu().numpy(), s_x.cpu().numpy(), rot.cpu().numpy()


def _check_rq(x_t, x32, perm, b):
    K = x32.shape[1]
    gq, gs, grot = _rq_gpu(x_t, perm, b)
    eq, es, erot = _rq_gpu(x_t, perm, b, clq.CLQ_CODES_E4M3)
    oq, os_, orot, oc = oracle.rotate_quant_act(x32, perm, b)
    check_rot(grot, orot)
    check_scales(gs, os_)
    check_codes(_codes(gq, K), oc, orot, os_)
    # both layouts carry the same codes and scales; the E4M3 path (for b >= 16
    # it reads each segment in an XOR order and restores the output signs)
    # gives the same rotation too
    assert np.array_equal(_codes(eq, K), _codes(gq, K)) and np.array_equal(es, gs)
    check_rot(erot, orot)
    if K % 128 == 0:  # the E2M3 layout (same XOR-ordered gather as E4M3)
        fq, fs, frot = _rq_gpu(x_t, perm, b, clq.CLQ_CODES_E2M3)
        assert fq.shape == (x32.shape[0], K // 4 * 3)
        assert np.array_equal(_codes(fq, K), _codes(gq, K)) and np.array_equal(fs, gs)
        check_rot(frot, orot)
    return gq, gs


# ------------------------------------------------------------ rotate-quant --
@pytest.mark.parametrize("b", [1, 2, 8, 16, 32, 64, 128, 256])
@pytest.mark.parametrize("dtype", ["f16", "bf16"])
def test_rotate_quant_block_sizes(b, dtype):
    K = 512
    x_t, x32 = _inputs(37, K, dtype, seed=b)
    _check_rq(x_t, x32, _perm(K, "random", b), b)


@pytest.mark.parametrize("M,K", [(1, 32), (3, 64), (17, 96), (64, 1152),
                                 (300, 1152), (33, 4608), (5, 12288),
                                 (9, 3072), (2, 16384)])
def test_rotate_quant_shapes(M, K):
    b = 32 if K % 64 else 64
    x_t, x32 = _inputs(M, K, "f16", seed=M + K)
    _check_rq(x_t, x32, _perm(K, "random", K), b)


@pytest.mark.parametrize("b,codes", [(64, clq.CLQ_CODES_E4M3), (64, clq.CLQ_CODES_E2M3),
                                     (128, clq.CLQ_CODES_E4M3), (32, clq.CLQ_CODES_E4M3),
                                     (64, clq.CLQ_CODES_INT4_PACKED)])
@pytest.mark.parametrize("with_rot", [False, True])
def test_rotate_quant_perm_4_byte_aligned(b, codes, with_rot):
    # The API asks perm for 4-byte alignment only; a perm 4 bytes past a
    # 16-byte boundary makes the kernels gather in natural order (no XOR
    # order, no sign restore).  Codes and scales must not change.
    M, K = 300, 1152
    x_t, x32 = _inputs(M, K, "f16", seed=b + 3)
    perm = _perm(K, "random", 19)
    X = x_t.to(DEV)
    buf = torch.zeros(K + 4, dtype=torch.int32, device=DEV)
    buf[1:K + 1] = torch.from_numpy(perm).to(DEV)
    pv = buf[1:K + 1]
    assert pv.data_ptr() % 16 == 4
    pa = torch.from_numpy(perm).to(DEV)
    ra = clq.rotate_quant_act(X, pa, b, codes, with_rot=with_rot)
    rb = clq.rotate_quant_act(X, pv, b, codes, with_rot=with_rot)
    torch.cuda.synchronize()
    assert torch.equal(ra[1], rb[1])
    assert np.array_equal(_codes(ra[0].cpu().numpy(), K), _codes(rb[0].cpu().numpy(), K))
    if with_rot:
        assert torch.equal(ra[2], rb[2])
    oq, os_, orot, oc = oracle.rotate_quant_act(x32, perm, b)
    check_scales(rb[1].cpu().numpy(), os_)
    check_codes(_codes(rb[0].cpu().numpy(), K), oc, orot, os_)


@pytest.mark.parametrize("K,b", [(1184, 32), (1216, 64), (1280, 128),
                                 (2112, 64)])
def test_rotate_quant_padding_lanes_do_not_leak(K, b):
    """K / 32 segments per row that do not fill whole warps: the CTA has
    padding lanes, which must not touch any row's abs-max.  Rows without
    outliers make any leak visible in the scales."""
    x_t, x32 = _inputs(45, K, "f16", seed=K, scale=0.02, outliers=0)
    _check_rq(x_t, x32, _perm(K, "random", K), b)


@pytest.mark.parametrize("kind", ["identity", "reversed", "random"])
def test_rotate_quant_permutations(kind):
    K = 1152
    x_t, x32 = _inputs(40, K, "f16", seed=7)
    _check_rq(x_t, x32, _perm(K, kind, 3), 64)


def test_rotate_quant_strided_rows():
    M, K, ld = 20, 256, 264
    big = torch.randn(M, ld, generator=torch.Generator().manual_seed(1)).half()
    view = big[:, :K]
    perm = _perm(K, "random", 5)
    g = clq.rotate_quant_act(view.to(DEV), torch.from_numpy(perm).to(DEV), 64,
                             with_rot=True)
    # the device view keeps the row stride of the padded buffer
    dev_big = big.to(DEV)
    g2 = clq.rotate_quant_act(dev_big[:, :K], torch.from_numpy(perm).to(DEV),
                              64, with_rot=True)
    torch.cuda.synchronize()
    assert dev_big[:, :K].stride(0) == ld
    oq, os_, orot, oc = oracle.rotate_quant_act(view.float().numpy(), perm, 64)
    for Xq, s, rot in (g, g2):
        check_rot(rot.cpu().numpy(), orot)
        check_codes(oracle.unpack_int4(Xq.cpu().numpy()), oc, orot, os_)


def test_rotate_quant_zero_rows_and_spikes():
    K, b = 256, 64
    x = np.zeros((6, K), np.float32)
    x[1, 5] = 3.0                        # single spike
    x[2, :] = 0.0                        # zero row
    x[3, ::b] = -2.0                     # one spike per block
    x[4, 7] = 65504.0                    # fp16 maximum
    x[5, :] = 1e-4
    x_t = torch.from_numpy(x).half()
    perm = _perm(K, "random", 9)
    gq, gs, grot = _rq_gpu(x_t, perm, b)
    oq, os_, orot, oc = oracle.rotate_quant_act(x_t.float().numpy(), perm, b)
    assert gs[0] == 0 and gs[2] == 0 and not gq[0].any() and not gq[2].any()
    check_rot(grot, orot)
    check_scales(gs, os_)
    assert np.array_equal(gq, oq)


@pytest.mark.parametrize("b", [64, 128])
def test_rotate_quant_hot_loops_edge_rows(b):
    # The E4M3 hot-path loops (wide at b = 64, paired at b = 128) on rows
    # with a zero row, single spikes, the bf16 maximum and values so small
    # that the row scale is subnormal in fp32 (scaled by 2^64 before the
    # reciprocal), against the oracle's codes and scales.
    K = 1152
    x = np.zeros((9, K), np.float32)
    x[1, 5] = 3.0
    x[3, ::b] = -2.0
    x[4, 7] = 3.3895314e38               # bf16 maximum
    x[5, :] = 1e-4
    x[6, :] = 3e-39                      # tiny rows with normal scales
    x[6, 11] = -5e-39
    x[7, 3] = 9e-41                      # one subnormal input: subnormal scale
    x[8] = np.random.default_rng(2).standard_normal(K).astype(np.float32) * 1e-38
    x_t = torch.from_numpy(x).to(torch.bfloat16)
    perm = _perm(K, "random", 29)
    eq, es, erot = _rq_gpu(x_t, perm, b, clq.CLQ_CODES_E4M3)
    Xq, s_x = clq.rotate_quant_act(x_t.to(DEV), torch.from_numpy(perm).to(DEV), b,
                                   clq.CLQ_CODES_E4M3)
    torch.cuda.synchronize()
    assert np.array_equal(s_x.cpu().numpy(), es)
    assert np.array_equal(_codes(Xq.cpu().numpy(), K), _codes(eq, K))
    oq, os_, orot, oc = oracle.rotate_quant_act(x_t.float().numpy(), perm, b)
    assert es[0] == 0 and es[2] == 0 and not _codes(eq, K)[0].any()
    assert 0 < es[7] < 1.17549435e-38    # the subnormal-scale path ran
    check_rot(erot, orot)
    check_scales(es, os_)
    check_codes(_codes(eq, K), oc, orot, os_)


def test_rotate_quant_exact_ties_half_even():
    # rotated rows with s = 1 exactly and entries at k + 1/2: X = X~ H / b.
    b, K = 16, 64
    rng = np.random.default_rng(3)
    rot = rng.integers(-6, 7, (8, K)).astype(np.float64) + 0.5
    rot[:, ::b] = 7.0                     # row abs-max 7 -> s = 1
    H = oracle.hadamard_sylvester(b).astype(np.float64)
    xp = (rot.reshape(8, K // b, b) @ H / b).reshape(8, K)
    perm = _perm(K, "random", 4)
    x = np.empty_like(xp)
    x[:, perm] = xp                       # X[:, perm[j]] = X_p[:, j]
    x_t = torch.from_numpy(x.astype(np.float32)).half()
    assert np.array_equal(x_t.float().numpy(), x.astype(np.float32))
    gq, gs, grot = _rq_gpu(x_t, perm, b)
    oq, os_, orot, oc = oracle.rotate_quant_act(x_t.float().numpy(), perm, b)
    assert np.array_equal(orot, rot.astype(np.float32))
    assert np.all(os_ == 1.0) and np.array_equal(gs, os_)
    assert np.array_equal(grot, orot)
    assert np.array_equal(gq, oq)         # ties to even, bit for bit


def test_rotate_quant_bad_perm_index_is_reported():
    K = 64
    x_t, _ = _inputs(4, K, "f16", seed=1)
    perm = _perm(K, "identity")
    perm[5] = K + 100
    clq.rotate_quant_act(x_t.to(DEV), torch.from_numpy(perm).to(DEV), 32)
    assert clq.device_status() == 7       # CLQ_ERR_DEVICE_INDEX
    assert clq.device_status() == 0       # read-and-clear


def test_prepare_weights_with_clip():
    N, K, b = 70, 1152, 64
    rng = np.random.default_rng(2)
    w = (rng.standard_normal((N, K)) * 0.02).astype(np.float32)
    w_t = torch.from_numpy(w).half()
    perm = _perm(K, "random", 1)
    _, _, orot0, _ = oracle.prepare_weights(w_t.float().numpy(), perm, b)
    clip = (np.max(np.abs(orot0), axis=1) * 0.6).astype(np.float32)
    clip[::3] = 1e9                        # no clipping on every third row
    Wq, s_w, rot = clq.prepare_weights(w_t.to(DEV), torch.from_numpy(perm).to(DEV),
                                       b, clip=torch.from_numpy(clip).to(DEV),
                                       with_rot=True)
    torch.cuda.synchronize()
    oq, os_, orot, oc = oracle.prepare_weights(w_t.float().numpy(), perm, b, clip)
    check_rot(rot.cpu().numpy(), orot)
    check_scales(s_w.cpu().numpy(), os_)
    check_codes(oracle.unpack_int4(Wq.cpu().numpy()), oc, orot, os_)


# -------------------------------------------------------------------- GEMM --
def test_expand_weights_is_exact_e4m3_of_codes():
    rng = np.random.default_rng(4)
    codes = rng.integers(-7, 8, (300, 1152)).astype(np.int8)
    codes[0, :16] = np.arange(-7, 9)[:16].clip(-7, 7)
    Wq = torch.from_numpy(oracle.pack_int4(codes)).to(DEV)
    We = clq.expand_weights(Wq)
    torch.cuda.synchronize()
    assert We.shape == (300, 1152)
    assert np.array_equal(_decode_e4m3(We.cpu().numpy()), codes.astype(np.float64))


def test_convert_codes_between_layouts():
    rng = np.random.default_rng(9)
    rows, K = 70, 1152
    codes = rng.integers(-7, 8, (rows, K)).astype(np.int8)
    codes[0, :15] = np.arange(-7, 8)
    packed = torch.from_numpy(oracle.pack_int4(codes)).to(DEV)
    e2 = clq.convert_codes(packed, K, clq.CLQ_CODES_E2M3)
    e4 = clq.convert_codes(e2, K, clq.CLQ_CODES_E4M3)
    back = clq.convert_codes(e4, K, clq.CLQ_CODES_INT4_PACKED)
    again = clq.convert_codes(e2, K, clq.CLQ_CODES_E2M3)
    torch.cuda.synchronize()
    assert np.array_equal(e2.cpu().numpy(), _encode_e2m3(codes))
    assert np.array_equal(_decode_e4m3(e4.cpu().numpy()), codes.astype(np.float64))
    assert torch.equal(back, packed) and torch.equal(again, e2)
    assert clq.device_status() == 0
    # packed -8 has no E2M3 encoding: written as 0 and reported
    bad = codes.copy()
    bad[3, 5] = -8
    e2b = clq.convert_codes(torch.from_numpy(oracle.pack_int4(bad)).to(DEV), K,
                            clq.CLQ_CODES_E2M3)
    assert clq.device_status() == 9           # CLQ_ERR_DEVICE_CODE
    fixed = bad.copy()
    fixed[3, 5] = 0
    assert np.array_equal(e2b.cpu().numpy(), _encode_e2m3(fixed))


def test_prepared_linear_keeps_one_weight_layout():
    rng = np.random.default_rng(3)
    N, K = 96, 1152
    W = torch.from_numpy((rng.standard_normal((N, K)) * 0.02).astype(np.float32)).half().to(DEV)
    perm = torch.from_numpy(_perm(K, "random", 2)).to(DEV)
    layer = clq.PreparedLinear.from_weight(W, perm, 64)
    # the default execution layout: E4M3, 1 B a weight plus scales and the swap vector
    assert layer.w_codes == clq.CLQ_CODES_E4M3 and layer.We.shape == (N, K)
    assert layer.resident_bytes() == N * K + 4 * N + 4 * K
    # on request E2M3, 0.75 B a weight
    small = clq.PreparedLinear.from_weight(W, perm, 64, w_codes=clq.CLQ_CODES_E2M3)
    assert small.We.shape == (N, K // 4 * 3)
    assert small.resident_bytes() == N * K * 3 // 4 + 4 * N + 4 * K
    Wq, s_w = clq.prepare_weights(W, perm, 64)
    X = torch.from_numpy(rng.standard_normal((40, K)).astype(np.float32)).half().to(DEV)
    torch.cuda.synchronize()
    assert torch.equal(layer.Wq, Wq) and torch.equal(small.Wq, Wq)
    assert torch.equal(layer.s_w, s_w) and torch.equal(small.s_w, s_w)
    Y = layer(X)
    assert torch.equal(Y, small(X))
    # packed-nibble weights (0.5 B a weight) with E4M3 or packed activations,
    # and packed activations with E4M3 weights: the same codes, so the same Y
    P, E = clq.CLQ_CODES_INT4_PACKED, clq.CLQ_CODES_E4M3
    for w_codes, a_codes in ((P, E), (P, P), (E, P)):
        lay = clq.PreparedLinear.from_weight(W, perm, 64, w_codes=w_codes, a_codes=a_codes)
        assert lay.act_codes == a_codes and lay.w_codes == w_codes
        if w_codes == P:
            assert lay.We.shape == (N, K // 2)
            assert lay.resident_bytes() == N * K // 2 + 4 * N + 4 * K
        assert torch.equal(lay.Wq, Wq)
        assert torch.equal(lay(X), Y)
    with pytest.raises(ValueError):
        clq.PreparedLinear.from_weight(W, perm, 64, w_codes=P, a_codes=clq.CLQ_CODES_E2M3)


def _gemm_case(M, N, K, b, dtype, seed, bias=True):
    x_t, x32 = _inputs(M, K, dtype, seed)
    rng = np.random.default_rng(seed + 1)
    w_t = torch.from_numpy((rng.standard_normal((N, K)) * 0.02).astype(np.float32)).to(TD[dtype])
    bias_t = (torch.from_numpy((rng.standard_normal(N) * 0.01).astype(np.float32)).to(TD[dtype])
              if bias else None)
    perm = _perm(K, "random", seed)
    oXq, os_x, _, _ = oracle.rotate_quant_act(x32, perm, b)
    oWq, os_w, _, _ = oracle.prepare_weights(w_t.float().numpy(), perm, b)
    b32 = None if bias_t is None else bias_t.float().numpy()
    y64, acc = oracle.w4a4_linear(oXq, os_x, oWq, os_w, b, b32)
    Wq = torch.from_numpy(oWq).to(DEV)
    Xq = torch.from_numpy(oXq).to(DEV)
    outs = []
    # every combination of storage (packed) and execution (E4M3) layouts, and
    # E2M3 with E2M3 (host-encoded from the oracle's codes)
    pairs = [(Xc, W) for Xc in (Xq, clq.expand_weights(Xq)) for W in (Wq, clq.expand_weights(Wq))]
    if K % 128 == 0:
        pairs.append((torch.from_numpy(_encode_e2m3(oracle.unpack_int4(oXq))).to(DEV),
                      torch.from_numpy(_encode_e2m3(oracle.unpack_int4(oWq))).to(DEV)))
    for Xc, W in pairs:
        Y, gacc = clq.w4a4_linear(Xc, torch.from_numpy(os_x).to(DEV), W,
                                  torch.from_numpy(os_w).to(DEV), b, K,
                                  None if bias_t is None else bias_t.to(DEV),
                                  out_dtype=TD[dtype], with_acc=True)
        torch.cuda.synchronize()
        assert np.array_equal(gacc.cpu().numpy(), acc)
        y = Y.float().cpu().numpy()
        check_output_elementwise(y, y64, acc, os_x, os_w, b, b32, dtype)
        check_output_frobenius(y, y64)
        outs.append(Y)
    for Y in outs[1:]:
        assert torch.equal(outs[0], Y)


@pytest.mark.parametrize("M,N,K", [(1, 1, 32), (3, 17, 64), (17, 64, 128),
                                   (64, 256, 1152), (300, 600, 1152),
                                   (129, 257, 96), (250, 1000, 160),
                                   (256, 512, 4608)])
def test_gemm_acc_exact_and_output(M, N, K):
    _gemm_case(M, N, K, 32, "f16", seed=M + N + K)


@pytest.mark.parametrize("dtype", ["f16", "bf16"])
def test_gemm_dtypes_and_no_bias(dtype):
    _gemm_case(200, 300, 1152, 64, dtype, seed=5, bias=False)
    _gemm_case(130, 260, 1152, 64, dtype, seed=6, bias=True)


@pytest.mark.parametrize("K", [1152, 4608, 12288, 16384])
def test_gemm_carrier_exact_at_extremes(K):
    """All codes +-7: |acc| reaches 49 K (602112 at K = 12288); mixed-sign
    rows make large partial sums cancel.  fp32 accumulation of the E4M3
    carrier must stay exact."""
    M, N = 136, 264
    rng = np.random.default_rng(K)
    qx = np.where(rng.random((M, K)) < 0.5, -7, 7).astype(np.int8)
    qw = np.where(rng.random((N, K)) < 0.5, -7, 7).astype(np.int8)
    qx[:8] = 7
    qw[:8] = 7
    qw[8:16] = -7
    qx[8:16, : K // 2] = 7
    qx[8:16, K // 2:] = -7                 # partial sums rise to 49 K/2, end at 0
    Xq = oracle.pack_int4(qx)
    Wq = oracle.pack_int4(qw)
    acc = oracle.int_gemm(qx, qw)
    ones_x = torch.ones(M, dtype=torch.float32, device=DEV)
    ones_w = torch.ones(N, dtype=torch.float32, device=DEV)
    Wd = torch.from_numpy(Wq).to(DEV)
    Xd = torch.from_numpy(Xq).to(DEV)
    pairs = [(Xc, W) for Xc in (Xd, clq.expand_weights(Xd)) for W in (Wd, clq.expand_weights(Wd))]
    pairs.append((torch.from_numpy(_encode_e2m3(qx)).to(DEV),
                  torch.from_numpy(_encode_e2m3(qw)).to(DEV)))
    for Xc, W in pairs:
        _, gacc = clq.w4a4_linear(Xc, ones_x, W, ones_w, 32, K,
                                  out_dtype=torch.bfloat16, with_acc=True)
        torch.cuda.synchronize()
        assert np.array_equal(gacc.cpu().numpy(), acc)


def test_gemm_random_codes_all_values():
    M, N, K = 160, 320, 2048
    rng = np.random.default_rng(11)
    qx = rng.integers(-7, 8, (M, K)).astype(np.int8)
    qw = rng.integers(-7, 8, (N, K)).astype(np.int8)
    acc = oracle.int_gemm(qx, qw)
    s = torch.ones(max(M, N), dtype=torch.float32, device=DEV)
    _, gacc = clq.w4a4_linear(torch.from_numpy(oracle.pack_int4(qx)).to(DEV), s[:M],
                              torch.from_numpy(oracle.pack_int4(qw)).to(DEV), s[:N], 32, K,
                              with_acc=True)
    torch.cuda.synchronize()
    assert np.array_equal(gacc.cpu().numpy(), acc)


# ------------------------------------------------------ end-to-end layers --
def _layer_e2e(cfg, li, M, rows=None):
    d = synth.layer_inputs(cfg, li, M=M)
    b = d["b"]
    calib = torch.from_numpy(d["calib"]).to(TD[d["dtype"]]).to(DEV)
    g_scores = clq.outlier_scores(calib)
    o_scores = oracle.outlier_scores(d["calib"])
    assert np.array_equal(g_scores.cpu().numpy(), o_scores)
    perm = clq.build_permutation(g_scores)
    assert np.array_equal(perm.numpy(), oracle.build_permutation(o_scores))
    permd = perm.to(DEV)
    layer = clq.PreparedLinear.from_weight(d["W"].to(DEV), permd, b, bias=d["bias"].to(DEV))
    X = d["X"].to(DEV)
    K = X.shape[1]
    Xq, s_x, rot = clq.rotate_quant_act(X, permd, b, with_rot=True)
    Y = clq.w4a4_linear(Xq, s_x, layer.Wq, layer.s_w, b, K, layer.bias, out_dtype=X.dtype)
    torch.cuda.synchronize()
    assert torch.equal(layer(X), Y)    # execution layouts (E4M3 codes) = storage
    rows = np.arange(M) if rows is None else rows
    p = perm.numpy()
    oWq, os_w, orot_w, owc = oracle.prepare_weights(d["W32"], p, b)
    check_scales(layer.s_w.cpu().numpy(), os_w)
    check_codes(oracle.unpack_int4(layer.Wq.cpu().numpy()), owc, orot_w, os_w)
    x32 = d["X32"][rows]
    oXq, os_x, orot, oc = oracle.rotate_quant_act(x32, p, b)
    check_rot(rot.cpu().numpy()[rows], orot)
    check_scales(s_x.cpu().numpy()[rows], os_x)
    check_codes(_codes(Xq.cpu().numpy()[rows], K), oc, orot, os_x)
    y64, _ = oracle.w4a4_linear(oXq, os_x, oWq, os_w, b, d["bias32"])
    check_output_frobenius(Y.float().cpu().numpy()[rows], y64)
    Yf = layer(X, fused=True)
    # the E2M3 execution layout on both sides of the GEMM
    l6 = clq.PreparedLinear.from_weight(d["W"].to(DEV), permd, b, bias=d["bias"].to(DEV),
                                        w_codes=clq.CLQ_CODES_E2M3)
    Y6 = l6(X)
    torch.cuda.synchronize()
    assert torch.equal(Yf, Y)          # fused = separate kernels, bit for bit
    assert torch.equal(Y6, Y)
    return d, layer, Y


def test_single_layer_full():
    _layer_e2e(synth.WORKLOADS["single_1152"], 0, 256)


@pytest.mark.parametrize("name", ["pixart_1024", "video_16x32x32", "mmdit_4608"])
def test_layer_sets_full_size_sampled_rows(name):
    cfg = synth.WORKLOADS[name]
    rng = np.random.default_rng(0)
    for li in range(len(cfg["layers"])):
        M = cfg["M"]
        rows = np.sort(np.concatenate([rng.choice(M, 40, replace=False),
                                       [0, M - 1]]))
        _layer_e2e(cfg, li, M, rows)


def test_video_token_permutation_equivariance():
    cfg = synth.WORKLOADS["video_16x32x32"]
    d, layer, Y = _layer_e2e(cfg, 0, cfg["M"], rows=np.arange(0, cfg["M"], 997))
    X2 = synth.temporal_reorder(d["X"]).to(DEV)
    Y2 = layer(X2)
    torch.cuda.synchronize()
    Y_re = synth.temporal_reorder(Y.cpu())
    assert torch.equal(Y2.cpu(), Y_re)


def test_prepared_linear_state_roundtrip(tmp_path):
    cfg = synth.WORKLOADS["single_1152"]
    d = synth.layer_inputs(cfg, 0, M=64)
    perm = torch.from_numpy(oracle.build_permutation(oracle.outlier_scores(d["calib"])))
    layer = clq.PreparedLinear.from_weight(d["W"].to(DEV), perm, 64, bias=d["bias"].to(DEV))
    torch.save(layer.state_dict(), tmp_path / "l.pt")
    layer2 = clq.PreparedLinear.from_state_dict(torch.load(tmp_path / "l.pt"))
    X = d["X"].to(DEV)
    assert torch.equal(layer(X), layer2(X))


# ------------------------------------------------------------------- fused --
@pytest.mark.parametrize("M,N,K,b,dtype", [(1, 16, 64, 32, "f16"), (3, 17, 96, 32, "f16"),
                                           (200, 300, 1152, 64, "f16"),
                                           (300, 600, 1152, 128, "bf16"),
                                           (129, 264, 4608, 256, "f16"),
                                           (64, 256, 12288, 128, "bf16"),
                                           (40, 128, 16384, 64, "f16"),
                                           # the widest rows of the concurrent form
                                           # (one row a tile) and the first K of
                                           # the sequential form with E4M3 weights
                                           (130, 200, 9216, 128, "f16"),
                                           (70, 130, 9248, 32, "bf16")])
def test_fused_matches_separate_and_oracle(M, N, K, b, dtype):
    x_t, x32 = _inputs(M, K, dtype, seed=M + K)
    rng = np.random.default_rng(K)
    w_t = torch.from_numpy((rng.standard_normal((N, K)) * 0.02).astype(np.float32)).to(TD[dtype])
    bias_t = torch.from_numpy((rng.standard_normal(N) * 0.01).astype(np.float32)).to(TD[dtype])
    perm = torch.from_numpy(_perm(K, "random", M))
    layer = clq.PreparedLinear.from_weight(w_t.to(DEV), perm.to(DEV), b, bias=bias_t.to(DEV))
    X = x_t.to(DEV)
    Y_sep = layer(X)
    ws = clq.fused_workspace(M, K, DEV)
    # the execution layout (E4M3), packed, and E2M3 where K % 128 == 0
    Ws = [layer.We, layer.Wq]
    if K % 128 == 0:
        Ws.append(clq.convert_codes(layer.We, K, clq.CLQ_CODES_E2M3))
    for W in Ws:
        Y_f = clq.fused_linear(X, layer.perm, b, W, layer.s_w, layer.bias, workspace=ws)
        torch.cuda.synchronize()
        assert torch.equal(Y_f, Y_sep)
    Y_again = clq.fused_linear(X, layer.perm, b, layer.We, layer.s_w, layer.bias, workspace=ws)
    assert torch.equal(Y_again, Y_sep)   # workspace reuse
    oWq, os_w, _, _ = oracle.prepare_weights(w_t.float().numpy(), perm.numpy(), b)
    y64 = oracle.fused_linear(x32, perm.numpy(), b, oWq, os_w, bias_t.float().numpy())
    check_output_frobenius(Y_sep.float().cpu().numpy(), y64)


def test_fused_small_workspace_rejected():
    X = torch.zeros((8, 64), dtype=torch.float16, device=DEV)
    perm = torch.arange(64, dtype=torch.int32, device=DEV)
    W = torch.zeros((16, 32), dtype=torch.uint8, device=DEV)
    s_w = torch.ones(16, device=DEV)
    small = torch.empty(64, dtype=torch.uint8, device=DEV)
    with pytest.raises(clq.ClqError) as e:
        clq.fused_linear(X, perm, 32, W, s_w, workspace=small)
    assert e.value.status == 1


# ------------------------------------------------------- failure handling --
def test_bounded_wait_selftest_reports_timeout():
    clq.selftest_bounded_wait(2_000_000)   # 2 ms
    assert clq.device_status() == 6        # CLQ_ERR_TIMEOUT
    # the context stays usable
    x_t, x32 = _inputs(8, 64, "f16", seed=3)
    _check_rq(x_t, x32, _perm(64, "random", 1), 32)
    assert clq.device_status() == 0


def test_empty_inputs_are_noops():
    z = torch.empty((0, 64), dtype=torch.float16, device=DEV)
    perm = torch.arange(64, dtype=torch.int32, device=DEV)
    Xq, s_x = clq.rotate_quant_act(z, perm, 32)
    assert Xq.shape == (0, 32) and s_x.shape == (0,)
    Wq = torch.zeros((0, 32), dtype=torch.uint8, device=DEV)
    Y = clq.w4a4_linear(Xq, s_x, Wq, torch.empty(0, device=DEV), 32, 64)
    assert Y.shape == (0, 0)
