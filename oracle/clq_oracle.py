"""CPU oracle for the CLQ W4A4 orthogonal-based-smoothing (OBS) linear layer.

TEST INFRASTRUCTURE ONLY.  Nothing in the product path may import or call this
module: only ``tests/``, ``__graft_entry__.smoke()`` and the ``cpu_baseline`` /
``--impl reference`` legs of ``bench.py`` use it.  It shares no code with the
CUDA path and takes every input as a plain array.

Each function restates one step of the method (arxiv 2509.24416) in the
paper's order, in plain numpy, slowly and without blocking or fusion:

* Sec. 3.3 "Data Preparing": batch mean S of the calibration activations.
* Sec. 3.3 "Outlier Detection": per-channel absolute maximum of S as the
  outlier score (Sec. 4.4's alternative metrics too); the top 50% of
  channels are moved to the left side.
* Sec. 3.3 "Orthogonal Smoothing" / "Overhead Analysis": G = S_swap H with H a
  block-diagonal +-1 Hadamard matrix; G is absorbed into the weights before
  quantization; the activations are rotated online; only the index vector s
  of the column swap is stored.
* Sec. 3.1, Eq. 1 with dynamic (per-input) activation bounds: uniform
  quantization to n = 4 bits, read here in its symmetric form l = -r.
* The INT4 x INT4 product, accumulated exactly in int64, then dequantized in
  fp64 with the bias added.
* Sec. 4.1's other bit settings (W4A8, W8A8): the same symmetric grid at
  8 bits and the same exact product (quant_linear, obs_linear).
* Eq. 1 itself for activations, asymmetric with the row's min and max as
  dynamic bounds, and the product of the dequantized operands (asym_linear).
* Sec. 3.4 / Eq. 3: the per-layer clip search over one percentile p of the
  rotated weights' magnitudes (clip_search).

Readings of the paper that this file fixes (the paper leaves them open):

1. Permutation direction.  The swap vector s holds, at position k, the index
   of the original column placed there (Sec. 3.3), so X_p[:, k] = X[:, s[k]].
2. Within-half order.  The paper needs no full descending order (Sec. 3.3);
   we rank channels by score descending with ties to the lower index, take the
   first floor(K/2) as the high set, and list the high set then the low set,
   each in ascending channel index.
3. Hadamard construction.  Sylvester, natural order:
   H_b[i, j] = (-1)^popcount(i & j), entries +-1 (Sec. 3.3), b a power of two.
   Blocks of size b tile the row; the 50/50 split need not fall on a block
   boundary.
4. Normalization.  H is kept unnormalized (exact +-1 arithmetic); since
   H_b H_b^T = b I, the product of rotated operands is divided by b once in
   the epilogue, which is exact (b is a power of two).
5. Symmetric 4-bit grid.  Eq. 1 with l = -r and qmax = 2^(n-1) - 1 = 7:
   r = max |row| (dynamic for activations, Sec. 3.1; optionally clipped for
   weights), s = r / 7 in fp32, q = clamp(rint(v / s), -7, 7) with fp32
   division and round-half-to-even (Eq. 1 says "nearest" and leaves ties
   open).  A zero row gets s = 0 and all-zero codes.  Code -8 is unused.
6. Precision.  The rotation is evaluated in fp64 and rounded once to fp32.
   For fp16 inputs every partial sum of a block is a multiple of 2^-24 below
   2^24 in magnitude, so the fp64 sums are exact and the fp32 result is the
   correctly rounded exact rotation.  The batch mean for the outlier score is
   taken in fp32 (sequential sum over the batch, then one division), the same
   precision the GPU path uses, because it decides an integer permutation.
7. Packing.  Byte j of a packed row holds code 2j in its low nibble and code
   2j+1 in its high nibble, as 4-bit two's complement.
8. Outlier-metric variants.  Sec. 4.4 names percentile (1 %, 99 %), top-k
   mean (k = 1 %), range and peak-average ratio without formulas; read as
   in outlier_scores() (percentile: max(|P1|, |P99|) with linear
   interpolation; k = max(1, round-half-up(T / 100)); PAR = peak / mean of
   |S|), each in fp32 in a fixed order.
9. Bit widths.  The paper runs W4A4, W4A8 and W8A8 (Sec. 4.1); the grid of
   reading 5 generalizes to n bits as qmax = 2^(n-1) - 1 (7 or 127): codes in
   [-qmax, qmax], s = r / qmax, code -2^(n-1) unused.  The product of n-bit
   codes is the same exact integer sum, dequantized by the same epilogue.
10. Asymmetric activations.  Eq. 1 as printed returns
   Round((Clip(x, l, r) - l) / (r - l) (2^n - 1)) (r - l) / (2^n - 1), which
   drops the offset l; read as x^ = q D + l with D = (r - l) / (2^n - 1) and
   q in [0, 2^n - 1] (the usual asymmetric fake quantization, and the only
   reading under which x^ approximates x).  Dynamic bounds l = min, r = max
   of the rotated row (Sec. 3.1).  The ratio is taken in the printed order,
   ((x - l) / (r - l)) (2^n - 1), in fp32, rounded half to even.  A constant
   row (r = l) has D = 0 and all codes 0, so x^ = l exactly.
11. Per-layer clip search (Sec. 3.4, Eq. 3, with the target layer taken to
   be the layer itself, since Eq. 2's cross-layer target needs a model).
   Under the symmetric weight grid (reading 5) the bounds satisfy l = -r, so
   the grid over (l, r) collapses to one percentile p in [beta, gamma]
   (beta = 0, gamma = 0.01, Sec. 4.1), the same p for every output channel
   of a matrix (Sec. 4.1), with r_n(p) the floor(p K)-th largest |W~[n, :]|
   (0-based, so p = 0 is the row's absolute maximum: no clipping).  The
   objective is ||Y - Y^||_F^2 on calibration tokens, Y = X W^T + bias in
   fp64 and Y^ the quantized layer (rotate-quant of X, weights prepared with
   clip r(p)) in fp64.  The smallest error wins; ties go to the smaller p.
"""

import numpy as np

QMAX = 7  # 2^(n-1) - 1 for n = 4 bits (symmetric reading of Eq. 1)
BIT_WIDTHS = (4, 8)  # Sec. 4.1: W4A4, W4A8, W8A8


def qmax_for_bits(bits):
    """Largest code of the symmetric n-bit grid, 2^(n-1) - 1 (reading 9)."""
    if bits not in BIT_WIDTHS:
        raise ValueError("bit width must be 4 or 8")
    return 2 ** (bits - 1) - 1


# ---------------------------------------------------------------- Sec. 3.3 --
def hadamard_sylvester(b):
    """Sylvester Hadamard matrix of order b in natural order, int64 +-1.

    H[i, j] = (-1)^popcount(i & j).  Sec. 3.3 ("Orthogonal Smoothing" and the
    +-1 storage remark under "Overhead Analysis").
    """
    if b < 1 or (b & (b - 1)) != 0:
        raise ValueError("Hadamard order must be a power of two")
    idx = np.arange(b, dtype=np.int64)
    anded = idx[:, None] & idx[None, :]
    parity = np.zeros((b, b), dtype=np.int64)
    bit = 1
    while bit < b:
        parity ^= (anded & bit) != 0
        bit <<= 1
    return np.where(parity == 1, -1, 1).astype(np.int64)


OUTLIER_METRICS = ("absmax", "percentile", "topk_mean", "range", "par")
PERCENTILE_PAIR = (0.01, 0.99)  # Sec. 4.4 "Choice of Outlier Metric": (1 %, 99 %)


def batch_mean(calib):
    """Sec. 3.3 "Data Preparing": S = mean of X [B, T, K] over the batch axis
    (fp32, summed over b in order, then divided by B)."""
    calib = np.asarray(calib, dtype=np.float32)
    if calib.ndim != 3:
        raise ValueError("calibration data must be [B, T, K]")
    B = calib.shape[0]
    total = np.zeros(calib.shape[1:], dtype=np.float32)
    for bi in range(B):
        total = total + calib[bi]
    return total / np.float32(B)


def topk_count(T):
    """k of the top-k mean: 1 % of the tokens (Sec. 4.4), rounded half up,
    at least 1 (reading 8)."""
    return max(1, (int(T) + 50) // 100)


def _percentile_fp32(sorted_col, q):
    """Linear interpolation between order statistics, every step in fp32:
    pos = q * (T - 1), lo = floor(pos), v = v[lo] + (pos - lo) * (v[lo+1] - v[lo])
    (reading 8)."""
    T = sorted_col.shape[0]
    pos = np.float32(q) * np.float32(T - 1)
    lo = int(np.floor(pos))
    hi = min(lo + 1, T - 1)
    frac = np.float32(pos - np.float32(lo))
    d = np.float32(sorted_col[hi] - sorted_col[lo])
    return np.float32(sorted_col[lo] + np.float32(frac * d))


def outlier_scores(calib, metric="absmax"):
    """Outlier score per channel from calibration activations [B, T, K].

    Sec. 3.3 "Outlier Detection": the score of channel c is max over tokens
    of |S[:, c]| (the method's choice).  Sec. 4.4 "Choice of Outlier Metric"
    names four alternatives, read here (reading 8) as, per channel of S:
      percentile: max(|P1|, |P99|), P linear-interpolated order statistics;
      topk_mean:  the mean of the k = topk_count(T) largest |S[t, c]|, summed
                  from the largest down in fp32;
      range:      max_t S - min_t S;
      par:        peak-to-average ratio max_t |S| / (sum_t |S| / T), the sum
                  taken over t in order in fp32; 0 for an all-zero channel.
    All arithmetic in fp32 in the stated order: the scores decide an integer
    permutation, and the GPU takes the same steps.
    """
    if metric not in OUTLIER_METRICS:
        raise ValueError("unknown outlier metric %r" % (metric,))
    S = batch_mean(calib)
    T, K = S.shape
    A = np.abs(S)
    if metric == "absmax":
        return np.max(A, axis=0).astype(np.float32)
    if metric == "range":
        return (np.max(S, axis=0) - np.min(S, axis=0)).astype(np.float32)
    if metric == "par":
        total = np.zeros(K, dtype=np.float32)
        for t in range(T):
            total = total + A[t]
        mean = total / np.float32(T)
        peak = np.max(A, axis=0)
        out = np.zeros(K, dtype=np.float32)
        nz = mean > 0
        out[nz] = (peak[nz] / mean[nz]).astype(np.float32)
        return out
    if metric == "percentile":
        Ss = np.sort(S, axis=0)
        out = np.empty(K, dtype=np.float32)
        for c in range(K):
            lo = _percentile_fp32(Ss[:, c], PERCENTILE_PAIR[0])
            hi = _percentile_fp32(Ss[:, c], PERCENTILE_PAIR[1])
            out[c] = max(abs(lo), abs(hi))
        return out
    # topk_mean
    k = topk_count(T)
    As = -np.sort(-A, axis=0)  # descending per channel
    total = np.zeros(K, dtype=np.float32)
    for t in range(k):
        total = total + As[t]
    return (total / np.float32(k)).astype(np.float32)


def build_permutation(scores):
    """Column-swap vector s from outlier scores (Sec. 3.3, reading 2).

    Channels whose rank (score descending, ties to the lower index) is below
    floor(K/2) form the high-peak set, placed on the left; the rest go right.
    Each side lists its channels in ascending index.
    """
    scores = np.asarray(scores, dtype=np.float32)
    K = scores.shape[0]
    order = sorted(range(K), key=lambda c: (-float(scores[c]), c))
    high = sorted(order[: K // 2])
    low = sorted(order[K // 2:])
    return np.array(high + low, dtype=np.int32)


def rotate_fp64(X, perm, b):
    """X_p H_blk in fp64: gather columns by s, then multiply every length-b
    block of the row by H_b (Sec. 3.3, G = S H applied to the activation).

    Rows are independent; any float input dtype is widened exactly to fp64.
    """
    X = np.asarray(X).astype(np.float64)
    perm = np.asarray(perm, dtype=np.int64)
    M, K = X.shape
    if K % b != 0:
        raise ValueError("K must be a multiple of the Hadamard block size")
    Xp = X[:, perm]
    H = hadamard_sylvester(b).astype(np.float64)
    return (Xp.reshape(M, K // b, b) @ H).reshape(M, K)


def rotate(X, perm, b):
    """Rotated rows rounded once to fp32 (reading 6)."""
    return rotate_fp64(X, perm, b).astype(np.float32)


# ------------------------------------------------------------ Sec. 3.1 Eq.1 --
def quantize_symmetric(V, clip=None, bits=4):
    """Per-row symmetric n-bit quantization of fp32 rows (Eq. 1, readings 5
    and 9).

    Returns (codes int8 [R, K] in [-qmax, qmax], scales fp32 [R]), qmax = 7
    for 4 bits and 127 for 8.  ``clip`` (one fp32 bound per row, > 0)
    replaces the row's absolute maximum by min(absmax, clip); values beyond
    it saturate at +-qmax.
    """
    qmax = qmax_for_bits(bits)
    V = np.asarray(V, dtype=np.float32)
    amax = np.max(np.abs(V), axis=1).astype(np.float32)
    if clip is not None:
        amax = np.minimum(amax, np.asarray(clip, dtype=np.float32))
    scale = (amax / np.float32(qmax)).astype(np.float32)
    codes = np.zeros(V.shape, dtype=np.int8)
    nz = scale > 0
    if np.any(nz):
        ratio = (V[nz] / scale[nz][:, None]).astype(np.float32)
        codes[nz] = np.clip(np.rint(ratio), -qmax, qmax).astype(np.int8)
    scale = np.where(nz, scale, np.float32(0)).astype(np.float32)
    return codes, scale


def quantize_asymmetric(V, bits=4):
    """Per-row asymmetric n-bit quantization of fp32 rows with dynamic bounds
    (Eq. 1 with l = min, r = max of the row; Sec. 3.1; reading 10).

    Returns (codes int16 [R, K] in [0, 2^n - 1], delta fp32 [R], lo fp32 [R]);
    the dequantized row is delta * codes + lo.
    """
    if bits not in BIT_WIDTHS:
        raise ValueError("bit width must be 4 or 8")
    levels = np.float32(2 ** bits - 1)
    V = np.asarray(V, dtype=np.float32)
    lo = np.min(V, axis=1).astype(np.float32)
    hi = np.max(V, axis=1).astype(np.float32)
    span = (hi - lo).astype(np.float32)
    codes = np.zeros(V.shape, dtype=np.int16)
    nz = span > 0
    if np.any(nz):
        shifted = (V[nz] - lo[nz][:, None]).astype(np.float32)
        frac = (shifted / span[nz][:, None]).astype(np.float32)
        ratio = (frac * levels).astype(np.float32)
        codes[nz] = np.clip(np.rint(ratio), 0, levels).astype(np.int16)
    delta = np.where(nz, span / levels, np.float32(0)).astype(np.float32)
    return codes, delta, lo


def dequantize_asymmetric(codes, delta, lo):
    """x^ = delta * q + lo per row, in fp64 (reading 10)."""
    return (np.asarray(codes, np.float64) * np.asarray(delta, np.float64)[:, None]
            + np.asarray(lo, np.float64)[:, None])


def rotate_quant_act_asym(X, perm, b, bits=4):
    """Online activation path with asymmetric dynamic quantization: gather by
    s, block Hadamard, then Eq. 1 per token (reading 10).

    Returns (codes int16 [M, K] in [0, 2^n - 1], delta fp32 [M], lo fp32 [M],
    x_rot fp32 [M, K]).
    """
    x_rot = rotate(X, perm, b)
    codes, delta, lo = quantize_asymmetric(x_rot, bits)
    return codes, delta, lo, x_rot


def asym_linear(qx, delta, lo, qw, s_w, b, bias=None):
    """The product of dequantized asymmetric activations and symmetric
    weights, by definition: y = X^ W^T / b + bias with X^ = delta q_x + lo
    and W^ = s_w q_w, all in fp64 (Sec. 3.3's G G^T = b I with the
    unnormalized H, reading 4)."""
    xh = dequantize_asymmetric(qx, delta, lo)
    wh = np.asarray(qw, np.float64) * np.asarray(s_w, np.float64)[:, None]
    y = xh @ wh.T / float(b)
    if bias is not None:
        y = y + np.asarray(bias).astype(np.float64)[None, :]
    return y


def pack_int4(codes):
    """Two codes per byte, code 2j in the low nibble (reading 7)."""
    codes = np.asarray(codes, dtype=np.int8)
    if codes.shape[1] % 2:
        raise ValueError("row length must be even to pack")
    lo = codes[:, 0::2].astype(np.int16) & 0xF
    hi = codes[:, 1::2].astype(np.int16) & 0xF
    return (lo | (hi << 4)).astype(np.uint8)


def unpack_int4(packed):
    """Inverse of pack_int4: sign-extend each nibble."""
    packed = np.asarray(packed, dtype=np.uint8).astype(np.int16)
    lo = packed & 0xF
    hi = (packed >> 4) & 0xF
    lo = np.where(lo >= 8, lo - 16, lo)
    hi = np.where(hi >= 8, hi - 16, hi)
    out = np.empty((packed.shape[0], packed.shape[1] * 2), dtype=np.int8)
    out[:, 0::2] = lo
    out[:, 1::2] = hi
    return out


def rotate_quant_act(X, perm, b, bits=4):
    """Online activation path: gather by s, block Hadamard, dynamic per-token
    scale, codes, pack (Sec. 3.1 dynamic quantization + Sec. 3.3).

    Returns (Xq, s_x fp32 [M], x_rot fp32 [M, K], codes int8 [M, K]); Xq is
    the packed uint8 [M, K/2] for 4 bits and the codes themselves for 8.
    """
    x_rot = rotate(X, perm, b)
    codes, s_x = quantize_symmetric(x_rot, bits=bits)
    return (pack_int4(codes) if bits == 4 else codes), s_x, x_rot, codes


def prepare_weights(W, perm, b, clip=None, bits=4):
    """Offline weight path: absorb G into W (W~ = W_p H_blk, Sec. 3.3
    "Overhead Analysis"), then per-output-channel symmetric n-bit codes.

    W is [N, K] as in nn.Linear.  Returns (Wq, s_w fp32 [N], w_rot fp32
    [N, K], codes int8 [N, K]); Wq is packed uint8 [N, K/2] for 4 bits and
    the codes themselves for 8.
    """
    w_rot = rotate(W, perm, b)
    codes, s_w = quantize_symmetric(w_rot, clip, bits=bits)
    return (pack_int4(codes) if bits == 4 else codes), s_w, w_rot, codes


# ------------------------------------------------------------ INT4 product --
def int_gemm(qx, qw):
    """acc[i, n] = sum_k qx[i, k] * qw[n, k], exact in int64."""
    acc = np.asarray(qx, dtype=np.int64) @ np.asarray(qw, dtype=np.int64).T
    if acc.size and np.max(np.abs(acc)) >= 2 ** 31:
        raise OverflowError("accumulator exceeds int32")
    return acc


def dequant_epilogue(acc, s_x, s_w, b, bias=None):
    """y = acc * s_x[i] * s_w[n] / b + bias[n] in fp64 (reading 4)."""
    y = (np.asarray(acc, dtype=np.float64)
         * np.asarray(s_x, dtype=np.float64)[:, None]
         * np.asarray(s_w, dtype=np.float64)[None, :] / float(b))
    if bias is not None:
        y = y + np.asarray(bias).astype(np.float64)[None, :]
    return y


def w4a4_linear(Xq, s_x, Wq, s_w, b, bias=None):
    """Packed INT4 x INT4 product with the dequant + bias epilogue.

    Returns (y fp64 [M, N], acc int64 [M, N]).
    """
    acc = int_gemm(unpack_int4(Xq), unpack_int4(Wq))
    return dequant_epilogue(acc, s_x, s_w, b, bias), acc


def quant_linear(qx, s_x, qw, s_w, b, bias=None):
    """Product of unpacked n-bit codes (any of W4A4, W4A8, W8A8) with the
    dequant + bias epilogue.  Returns (y fp64 [M, N], acc int64 [M, N])."""
    acc = int_gemm(qx, qw)
    return dequant_epilogue(acc, s_x, s_w, b, bias), acc


def obs_linear(X, perm, b, qw, s_w, bias=None, a_bits=4):
    """The layer at any bit setting: rotate-quant of X to a_bits, then the
    product with the prepared weight codes qw (int8 [N, K], any width)."""
    _, s_x, _, qx = rotate_quant_act(X, perm, b, bits=a_bits)
    y, _ = quant_linear(qx, s_x, qw, s_w, b, bias)
    return y


def fused_linear(X, perm, b, Wq, s_w, bias=None):
    """Rotate-quant of X followed by the W4A4 product (same arithmetic as the
    two separate steps; the fusion is a GPU scheduling choice only)."""
    Xq, s_x, _, _ = rotate_quant_act(X, perm, b)
    y, _ = w4a4_linear(Xq, s_x, Wq, s_w, b, bias)
    return y


def linear_fp64(X, W, bias=None):
    """Unquantized X W^T + bias in fp64, for reporting quantization error."""
    y = np.asarray(X).astype(np.float64) @ np.asarray(W).astype(np.float64).T
    if bias is not None:
        y = y + np.asarray(bias).astype(np.float64)[None, :]
    return y


# --------------------------------------------- Sec. 3.4 Eq. 3 clip search --
CLIP_BETA, CLIP_GAMMA = 0.0, 0.01  # Sec. 4.1: beta = 0, gamma = 0.01


def clip_grid(G, beta=CLIP_BETA, gamma=CLIP_GAMMA):
    """G evenly spaced percentiles from beta to gamma (fp64)."""
    if G < 1:
        raise ValueError("grid needs at least one point")
    if G == 1:
        return np.array([beta], dtype=np.float64)
    return beta + (gamma - beta) * np.arange(G, dtype=np.float64) / (G - 1)


def clip_rank(p, K):
    """0-based rank, from the top, of the clip bound at percentile p
    (reading 11): floor(p K)."""
    return int(np.floor(float(p) * K))


def clip_table(w_rot, J):
    """The J largest |w_rot[n, k]| of every row, largest first (fp32)."""
    A = np.abs(np.asarray(w_rot, dtype=np.float32))
    return -np.sort(-A, axis=1)[:, :J]


def clip_search(X, W, perm, b, bias=None, grid=None):
    """Eq. 3 per layer (reading 11): for every percentile p of the grid, clip
    each output channel of W~ at r_n(p), quantize, run the W4A4 layer on the
    calibration tokens X and measure ||Y - Y^||_F^2 against the fp64 layer.

    Returns (errors fp64 [G], best grid index, clip fp32 [N] of the best p,
    grid fp64 [G]).
    """
    grid = clip_grid(11) if grid is None else np.asarray(grid, np.float64)
    W = np.asarray(W)
    K = W.shape[1]
    w_rot = rotate(W, perm, b)
    J = max(clip_rank(p, K) for p in grid) + 1
    table = clip_table(w_rot, J)
    Y = linear_fp64(X, W, bias)
    errors = np.empty(len(grid), dtype=np.float64)
    clips = []
    for g, p in enumerate(grid):
        clip = table[:, clip_rank(p, K)].astype(np.float32)
        Wq, s_w, _, _ = prepare_weights(W, perm, b, clip)
        Yh = fused_linear(X, perm, b, Wq, s_w, bias)
        errors[g] = float(np.sum((Y - Yh) ** 2))
        clips.append(clip)
    best = int(np.argmin(errors))  # first minimum: ties to the smaller p
    return errors, best, clips[best], grid
