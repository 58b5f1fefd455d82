"""GPU parity for asymmetric activation quantization (Eq. 1 with the row's
min and max as dynamic bounds, Sec. 3.1) and its zero-point epilogue,
against the oracle.

Tolerances (in addition to tests/parity_utils.py):
* lo (row minimum) and delta = (max - min) / (2^n - 1) come from the GPU's
  rotated row, whose elements carry at most ~log2(b) roundings: |lo_g - lo_o|
  <= 1e-5 max_k |X~[i, k]|, and |delta_g - delta_o| <= 2.5e-7 delta_o +
  2e-5 max_k |X~[i, k]| / (2^n - 1).
* codes: equal, except off by one where the oracle's ratio
  (X~ - l) / (r - l) (2^n - 1) lies within 1e-4 of a half-integer.
* outputs: with the oracle's codes, |Y - y64| <= u |y64| + 1e-6 (|delta acc
  s_w / b| + |m wsum s_w / b| + |bias|) + tiny, the two epilogue terms
  counted separately because they can cancel.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2509_24416_gb300 import clq, synth
from parity_utils import check_output_frobenius, check_rot

pytestmark = pytest.mark.gpu
DEV = torch.device("cuda:0")
TD = {"f16": torch.float16, "bf16": torch.bfloat16}
E4M3, SPLIT, PACKED = clq.CLQ_CODES_E4M3, clq.CLQ_CODES_E4M3_SPLIT, clq.CLQ_CODES_INT4_PACKED


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
    """E4M3 byte of integers the format holds exactly."""
    v = np.asarray(v, np.int64)
    a = np.abs(v).astype(np.float64)
    f, x = np.frexp(np.where(a == 0, 1.0, a))
    m = (f * 2 - 1) * 8
    assert np.array_equal(m, np.rint(m)), "not an E4M3 value"
    byte = ((x - 1 + 7) << 3) | m.astype(np.int64)
    return (np.where(a == 0, 0, byte) | np.where(v < 0, 0x80, 0)).astype(np.uint8)


def _to_layout(c, layout):
    c = np.asarray(c, np.int64)
    if layout == E4M3:
        return _encode_e4m3_int(c)
    if layout == PACKED:
        return oracle.pack_int4(c.astype(np.int8))
    h = np.floor_divide(c + 8, 16)
    return np.concatenate([_encode_e4m3_int(16 * h), _encode_e4m3_int(c - 16 * h)], axis=1)


def _from_layout(Q, layout, K):
    Q = np.asarray(Q)
    if layout == PACKED:
        return oracle.unpack_int4(Q).astype(np.int64)
    if layout == E4M3:
        v = _decode_e4m3(Q)
        assert np.array_equal(v, np.rint(v))
        return v.astype(np.int64)
    v = _decode_e4m3(Q[:, :K]) + _decode_e4m3(Q[:, K:])
    return v.astype(np.int64)


def _check_asym(gq, gdelta, glo, oq, odelta, olo, orot, bits):
    top = 2 ** bits - 1
    rowmax = np.max(np.abs(orot), axis=1)
    assert np.all(np.abs(glo - olo) <= 1e-5 * rowmax)
    assert np.all(np.abs(gdelta.astype(np.float64) - odelta)
                  <= 2.5e-7 * odelta + 2e-5 * rowmax / top)
    assert gq.min() >= 0 and gq.max() <= top
    bad = gq != oq
    n_bad = int(np.count_nonzero(bad))
    if n_bad:
        assert np.all(np.abs(gq[bad] - oq[bad]) == 1)
        span = (odelta * top).astype(np.float64)[:, None] * np.ones_like(orot, np.float64)
        lo = olo.astype(np.float64)[:, None] * np.ones_like(orot, np.float64)
        ratio = (orot.astype(np.float64)[bad] - lo[bad]) / span[bad] * top
        assert np.all(np.abs(np.abs(ratio - np.floor(ratio)) - 0.5) <= 1e-4)
        assert n_bad <= max(1, int(1e-4 * gq.size)), n_bad
    return n_bad


def _inputs(M, K, dtype, seed, offset=0.0):
    rng = np.random.default_rng(seed)
    x = rng.standard_normal((M, K)).astype(np.float32) * 2.0 + offset
    ch = rng.choice(K, min(4, K), replace=False)
    x[:, ch] *= 30
    t = torch.from_numpy(x).to(TD[dtype])
    return t, t.float().numpy()


@pytest.mark.parametrize("layout,bits", [(E4M3, 4), (PACKED, 4), (SPLIT, 8)])
@pytest.mark.parametrize("M,K,b,dtype", [(300, 1152, 64, "f16"), (77, 96, 32, "bf16"),
                                         (129, 4608, 128, "f16"), (40, 256, 1, "bf16")])
def test_rotate_quant_asym(layout, bits, M, K, b, dtype):
    x_t, x32 = _inputs(M, K, dtype, seed=M + K, offset=1.5)
    x_t[2] = 0.0           # rotates to a constant row: delta 0, every code 0
    x32[2] = 0.0
    perm = np.random.default_rng(K + 1).permutation(K).astype(np.int32)
    Xq, delta, lo, rot = clq.rotate_quant_act_asym(x_t.to(DEV), torch.from_numpy(perm).to(DEV),
                                                   b, codes=layout, with_rot=True)
    torch.cuda.synchronize()
    oq, od, olo, orot = oracle.rotate_quant_act_asym(x32, perm, b, bits)
    check_rot(rot.cpu().numpy(), orot)
    gq = _from_layout(Xq.cpu().numpy(), layout, K) + 2 ** (bits - 1)
    _check_asym(gq, delta.cpu().numpy(), lo.cpu().numpy(), oq, od, olo, orot, bits)
    assert delta[2].item() == 0.0 and np.all(gq[2] == 0)


def test_rotate_quant_asym_edge_rows():
    # asymmetric E4M3 codes at b = 64 (the wide loop): a zero row, a
    # constant row, spikes up to 1e38, and a row whose span is subnormal in
    # fp32 (exact divisions), against the oracle.
    K, b = 1152, 64
    x = np.zeros((7, K), np.float32)     # row 0 rotates to zeros: span 0
    x[1, :] = 2.5                        # constant row: one nonzero output a block
    x[2, 5] = 3.0
    x[3, 7] = -1e38                      # near the top of bf16, span still finite
    x[4, 3] = 9e-41                      # span subnormal
    x[5] = np.random.default_rng(4).standard_normal(K).astype(np.float32) + 7.0
    x[6, ::b] = -2.0
    x_t = torch.from_numpy(x).to(torch.bfloat16)
    perm = np.random.default_rng(31).permutation(K).astype(np.int32)
    Xq, delta, lo, rot = clq.rotate_quant_act_asym(x_t.to(DEV), torch.from_numpy(perm).to(DEV),
                                                   b, codes=E4M3, with_rot=True)
    Xq2, delta2, lo2 = clq.rotate_quant_act_asym(x_t.to(DEV), torch.from_numpy(perm).to(DEV),
                                                 b, codes=E4M3)
    torch.cuda.synchronize()
    assert torch.equal(delta, delta2) and torch.equal(lo, lo2)
    gq = _from_layout(Xq.cpu().numpy(), E4M3, K) + 8
    assert np.array_equal(gq, _from_layout(Xq2.cpu().numpy(), E4M3, K) + 8)
    oq, od, olo, orot = oracle.rotate_quant_act_asym(x_t.float().numpy(), perm, b, 4)
    assert 0 < delta[4].item() < 1.17549435e-38     # the exact-division path ran
    assert delta[0].item() == 0.0 and np.all(gq[0] == 0)
    check_rot(rot.cpu().numpy(), orot)
    _check_asym(gq, delta.cpu().numpy(), lo.cpu().numpy(), oq, od, olo, orot, 4)


@pytest.mark.parametrize("layout,bits", [(E4M3, 4), (SPLIT, 8)])
@pytest.mark.parametrize("with_rot", [False, True])
def test_rotate_quant_asym_perm_4_byte_aligned(layout, bits, with_rot):
    # perm 4 bytes past a 16-byte boundary: natural-order gather, no sign
    # restore; the codes, steps and minima must equal the aligned run's.
    M, K, b = 300, 1152, 64
    x_t, x32 = _inputs(M, K, "bf16", seed=5, offset=1.5)
    perm = np.random.default_rng(23).permutation(K).astype(np.int32)
    X = x_t.to(DEV)
    buf = torch.zeros(K + 4, dtype=torch.int32, device=DEV)
    buf[1:K + 1] = torch.from_numpy(perm).to(DEV)
    pv = buf[1:K + 1]
    assert pv.data_ptr() % 16 == 4
    ra = clq.rotate_quant_act_asym(X, torch.from_numpy(perm).to(DEV), b, codes=layout,
                                   with_rot=with_rot)
    rb = clq.rotate_quant_act_asym(X, pv, b, codes=layout, with_rot=with_rot)
    torch.cuda.synchronize()
    assert torch.equal(ra[1], rb[1]) and torch.equal(ra[2], rb[2])
    ga = _from_layout(ra[0].cpu().numpy(), layout, K)
    gb = _from_layout(rb[0].cpu().numpy(), layout, K)
    assert np.array_equal(ga, gb)
    if with_rot:
        assert torch.equal(ra[3], rb[3])
    oq, od, olo, orot = oracle.rotate_quant_act_asym(x32, perm, b, bits)
    _check_asym(gb + 2 ** (bits - 1), rb[1].cpu().numpy(), rb[2].cpu().numpy(), oq, od, olo,
                orot, bits)


@pytest.mark.parametrize("layout,bits", [(PACKED, 4), (E4M3, 4), (SPLIT, 8)])
def test_weight_code_sums(layout, bits):
    N, K = 300, 1152
    rng = np.random.default_rng(bits)
    top = 7 if bits == 4 else 127
    q = rng.integers(-top, top + 1, (N, K))
    q[0] = top
    q[1] = -top
    W = torch.from_numpy(_to_layout(q, layout)).to(DEV)
    wsum = clq.weight_code_sums(W, K)
    torch.cuda.synchronize()
    assert np.array_equal(wsum.cpu().numpy(), q.sum(axis=1).astype(np.float32))


def _asym_product(qx, d, lo, qw, s_w, b, a_bits, w_bits, dtype, bias):
    M, K = qx.shape
    half = 2 ** (a_bits - 1)
    c = qx - half
    Xq = torch.from_numpy(_to_layout(c, SPLIT if a_bits == 8 else E4M3)).to(DEV)
    W = torch.from_numpy(_to_layout(qw, SPLIT if w_bits == 8 else E4M3)).to(DEV)
    wsum = clq.weight_code_sums(W, K)
    bias_t = torch.from_numpy(bias).to(TD[dtype]).to(DEV)
    b32 = bias_t.float().cpu().numpy()
    Y, gacc = clq.linear_asym(Xq, torch.from_numpy(d).to(DEV), torch.from_numpy(lo).to(DEV), W,
                              torch.from_numpy(s_w).to(DEV), wsum, b, K, bias_t,
                              out_dtype=TD[dtype], with_acc=True)
    torch.cuda.synchronize()
    y64 = oracle.asym_linear(qx, d, lo, qw, s_w, b, b32)
    assert np.array_equal(gacc.cpu().numpy(), oracle.int_gemm(c, qw))
    acc = oracle.int_gemm(c, qw).astype(np.float64)
    m = lo.astype(np.float64) + half * d.astype(np.float64)
    ws = qw.sum(axis=1).astype(np.float64)
    t1 = np.abs(acc * d[:, None] * s_w[None, :] / b)
    t2 = np.abs(m[:, None] * ws[None, :] * s_w[None, :] / b)
    u = 2.0 ** -11 if dtype == "f16" else 2.0 ** -8
    tiny = 2.0 ** -24 if dtype == "f16" else 2.0 ** -126
    y = Y.float().cpu().numpy()
    tol = u * np.abs(y64) + 1e-6 * (t1 + t2 + np.abs(b32)[None, :]) + tiny
    assert np.all(np.abs(y - y64) <= tol), float(np.max(np.abs(y - y64) - tol))
    return y, y64


@pytest.mark.parametrize("a_bits,w_bits", [(4, 4), (8, 4), (8, 8)])
@pytest.mark.parametrize("M,N,K", [(1, 1, 32), (17, 64, 128), (300, 600, 1152),
                                   (129, 257, 96), (256, 512, 4608)])
def test_linear_asym_against_definition(a_bits, w_bits, M, N, K):
    rng = np.random.default_rng(M + N + K + a_bits + w_bits)
    qx = rng.integers(0, 2 ** a_bits, (M, K))
    wt = 2 ** (w_bits - 1) - 1
    qw = rng.integers(-wt, wt + 1, (N, K))
    d = rng.uniform(0.01, 0.1, M).astype(np.float32)
    lo = rng.uniform(-2.0, 0.5, M).astype(np.float32)
    s_w = rng.uniform(0.001, 0.01, N).astype(np.float32)
    bias = (rng.standard_normal(N) * 0.1).astype(np.float32)
    for dtype in ("f16", "bf16"):
        y, y64 = _asym_product(qx, d, lo, qw, s_w, 32, a_bits, w_bits, dtype, bias)
        check_output_frobenius(y, y64)


@pytest.mark.parametrize("a_bits,w_bits", [(4, 4), (8, 4), (8, 8)])
def test_layer_asym_end_to_end(a_bits, w_bits):
    """The ffn_down layer of the PixArt set (post-GELU activations, all above
    -0.17): rotate-quant with asymmetric codes, then the zero-point product,
    against the oracle layer."""
    d = synth.layer_inputs(dict(synth.WORKLOADS["pixart_1024"], M=512), 3)
    b, K = d["b"], d["K"]
    td = TD[d["dtype"]]
    calib = torch.from_numpy(d["calib"]).to(td).to(DEV)
    perm = clq.build_permutation(clq.outlier_scores(calib))
    permd = perm.to(DEV)
    X = d["X"].to(DEV)
    layout_x = SPLIT if a_bits == 8 else E4M3
    layout_w = SPLIT if w_bits == 8 else E4M3
    Wq, s_w = clq.prepare_weights(d["W"].to(DEV), permd, b, codes=layout_w)
    wsum = clq.weight_code_sums(Wq, K)
    Xq, delta, lo = clq.rotate_quant_act_asym(X, permd, b, codes=layout_x)
    Y = clq.linear_asym(Xq, delta, lo, Wq, s_w, wsum, b, K, d["bias"].to(DEV), out_dtype=td)
    torch.cuda.synchronize()
    p = perm.numpy()
    oq, od, olo, orot = oracle.rotate_quant_act_asym(d["X32"], p, b, a_bits)
    gq = _from_layout(Xq.cpu().numpy(), layout_x, K) + 2 ** (a_bits - 1)
    _check_asym(gq, delta.cpu().numpy(), lo.cpu().numpy(), oq, od, olo, orot, a_bits)
    _, os_w, _, owc = oracle.prepare_weights(d["W32"], p, b, bits=w_bits)
    y64 = oracle.asym_linear(oq, od, olo, owc, os_w, b, d["bias32"])
    y = Y.float().cpu().numpy()
    check_output_frobenius(y, y64)


@pytest.mark.parametrize("li", [0, 3])
def test_pixart_layer_full_size_sampled_rows_asym(li):
    """Asymmetric W4A4 on a PixArt-1024 layer at its full 8192 tokens, 42
    sampled rows against the oracle."""
    cfg = synth.WORKLOADS["pixart_1024"]
    d = synth.layer_inputs(cfg, li)
    b, K = d["b"], d["K"]
    M = cfg["M"]
    rows = np.sort(np.concatenate([np.random.default_rng(li).choice(M, 40, replace=False),
                                   [0, M - 1]]))
    perm = oracle.build_permutation(oracle.outlier_scores(d["calib"]))
    permd = torch.from_numpy(perm).to(DEV)
    Wq, s_w = clq.prepare_weights(d["W"].to(DEV), permd, b, codes=E4M3)
    wsum = clq.weight_code_sums(Wq, K)
    Xq, delta, lo = clq.rotate_quant_act_asym(d["X"].to(DEV), permd, b, codes=E4M3)
    Y = clq.linear_asym(Xq, delta, lo, Wq, s_w, wsum, b, K, d["bias"].to(DEV),
                        out_dtype=TD[d["dtype"]])
    torch.cuda.synchronize()
    oq, od, olo, orot = oracle.rotate_quant_act_asym(d["X32"][rows], perm, b, 4)
    gq = _from_layout(Xq.cpu().numpy()[rows], E4M3, K) + 8
    _check_asym(gq, delta.cpu().numpy()[rows], lo.cpu().numpy()[rows], oq, od, olo, orot, 4)
    _, os_w, _, owc = oracle.prepare_weights(d["W32"], perm, b)
    y64 = oracle.asym_linear(oq, od, olo, owc, os_w, b, d["bias32"])
    check_output_frobenius(Y.float().cpu().numpy()[rows], y64)
