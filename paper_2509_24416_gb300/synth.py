"""Seeded synthetic inputs shaped like the DiT layers the paper quantizes.

The paper evaluates on PixArt-alpha and Open-Sora 1.2 (Sec. 4.1); neither the
weights nor the activations are available, so these generators stand in with
the layer shapes of those models and the activation structure the paper
describes (a few channels with large outliers, Sec. 1 and Sec. 3.3).  This
module holds only random-number generation and workload shaping (outlier
channels, GELU for the FFN down-projection input, text-token scaling); none
of the quantization method's arithmetic lives here.  Every draw comes from a
counter-based Philox generator with a fixed seed.
"""

import numpy as np
import torch

SEED_X, SEED_W, SEED_BIAS, SEED_CHANNELS, SEED_CALIB = 0, 1, 2, 3, 4


def _rng(seed):
    return np.random.Generator(np.random.Philox(seed))


def layer_seed(base, layer):
    return int(base) + 16 * int(layer)


def outlier_channels(K, count, lo, hi, seed, fixed_factor=None):
    """Pick ``count`` channels of K and a scale factor for each
    (U(lo, hi), or ``fixed_factor`` for all)."""
    g = _rng(seed)
    idx = np.sort(g.choice(K, size=count, replace=False)).astype(np.int64)
    if fixed_factor is not None:
        fac = np.full(count, float(fixed_factor), dtype=np.float32)
    else:
        fac = g.uniform(lo, hi, size=count).astype(np.float32)
    return idx, fac


def activations(M, K, channels, seed, gelu=False, text_rows=0,
                text_scale=1.0):
    """N(0, 1) tokens x channels with the given outlier channels scaled;
    optionally passed through exact-erf GELU (FFN down-projection input) and
    with the last ``text_rows`` rows scaled (MMDiT text tokens).  fp32."""
    g = _rng(seed)
    x = g.standard_normal((M, K), dtype=np.float32)
    idx, fac = channels
    x[:, idx] *= fac[None, :]
    if gelu:
        x = torch.nn.functional.gelu(torch.from_numpy(x)).numpy()
    if text_rows:
        x[M - text_rows:, :] *= np.float32(text_scale)
    return x


def calibration(B, T, K, channels, seed, gelu=False):
    """[B, T, K] calibration activations from the same distribution."""
    return np.stack([activations(T, K, channels, seed + 1000 * i, gelu)
                     for i in range(B)])


def normal(shape, std, seed):
    g = _rng(seed)
    return (g.standard_normal(shape, dtype=np.float32) * np.float32(std))


def to_torch(arr, dtype):
    """fp32 numpy -> CPU torch tensor in 'f16' or 'bf16' (round to nearest)."""
    td = {"f16": torch.float16, "bf16": torch.bfloat16}[dtype]
    return torch.from_numpy(np.ascontiguousarray(arr)).to(td)


def exact_f32(t):
    """The exact values of a low-precision tensor as fp32 numpy."""
    return t.detach().to("cpu", torch.float32).numpy()


# ----------------------------------------------------------------- workloads
# Layer shapes (K in, N out) of one DiT block: QKV, attention out, FFN up,
# FFN down.  The down projection's input is post-GELU.
PIXART_LAYERS = (("qkv", 1152, 3456), ("attn_out", 1152, 1152),
                 ("ffn_up", 1152, 4608), ("ffn_down", 4608, 1152))
MMDIT_LAYERS = (("qkv", 3072, 9216), ("attn_out", 3072, 3072),
                ("ffn_up", 3072, 12288), ("ffn_down", 12288, 3072))

WORKLOADS = {
    # X [256, 1152] with 8 channels x40, W N(0, 0.02^2), b = 64, fp16.
    "single_1152": dict(M=256, layers=(("linear", 1152, 1152),), b=64,
                        dtype="f16", out_frac=None, out_count=8,
                        out_lo=40.0, out_hi=40.0, w_std=0.02,
                        text_rows=0, text_scale=1.0),
    # PixArt-alpha block at 1024px: 2 x 4096 tokens, hidden 1152, b = 64.
    "pixart_1024": dict(M=8192, layers=PIXART_LAYERS, b=64, dtype="f16",
                        out_frac=0.01, out_count=None, out_lo=20.0,
                        out_hi=60.0, w_std=0.02, text_rows=0,
                        text_scale=1.0),
    # Video DiT: 16 frames x 32 x 32 patches = 16384 tokens, b = 128, bf16.
    "video_16x32x32": dict(M=16384, layers=PIXART_LAYERS, b=128,
                           dtype="bf16", out_frac=0.01, out_count=None,
                           out_lo=20.0, out_hi=60.0, w_std=0.02,
                           text_rows=0, text_scale=1.0,
                           temporal=dict(frames=16, tokens_per_frame=1024)),
    # MMDiT: 4096 image + 512 text tokens, hidden 3072, b = 128, bf16.
    "mmdit_4608": dict(M=4608, layers=MMDIT_LAYERS, b=128, dtype="bf16",
                       out_frac=0.005, out_count=None, out_lo=50.0,
                       out_hi=100.0, w_std=0.015, text_rows=512,
                       text_scale=3.0),
}


def n_outliers(cfg, K):
    if cfg["out_count"] is not None:
        return int(cfg["out_count"])
    return int(round(cfg["out_frac"] * K))


def layer_inputs(cfg, li, M=None, calib_tokens=256, calib_batch=4, batch=0):
    """All seeded inputs of layer ``li`` of a workload, as numpy fp32 holding
    values already rounded to the workload dtype, plus the torch tensors.
    ``batch`` selects another token batch of the same distribution (the
    activations' seed moves; weights, bias and calibration do not), so that
    ranks of a multi-GPU run each process their own batch.

    Returns a dict with X, W, bias (torch, CPU, workload dtype), the exact
    fp32 copies X32, W32, bias32, and the calibration batch calib [B, T, K]
    (fp32 values rounded through the workload dtype).
    """
    name, K, N = cfg["layers"][li]
    M = cfg["M"] if M is None else M
    gelu = name == "ffn_down"
    ch = outlier_channels(K, n_outliers(cfg, K), cfg["out_lo"],
                          cfg["out_hi"], layer_seed(SEED_CHANNELS, li),
                          fixed_factor=(cfg["out_lo"]
                                        if cfg["out_lo"] == cfg["out_hi"]
                                        else None))
    dt = cfg["dtype"]
    X = to_torch(activations(M, K, ch, layer_seed(SEED_X, li) + 100003 * int(batch), gelu,
                             min(cfg["text_rows"], M), cfg["text_scale"]), dt)
    W = to_torch(normal((N, K), cfg["w_std"], layer_seed(SEED_W, li)), dt)
    bias = to_torch(normal((N,), 0.01, layer_seed(SEED_BIAS, li)), dt)
    cal = calibration(calib_batch, calib_tokens, K, ch,
                      layer_seed(SEED_CALIB, li), gelu)
    cal = exact_f32(to_torch(cal, dt))
    return dict(name=name, K=K, N=N, M=M, b=cfg["b"], dtype=dt, X=X, W=W,
                bias=bias, X32=exact_f32(X), W32=exact_f32(W),
                bias32=exact_f32(bias), calib=cal)


def temporal_reorder(X, frames=16, tokens_per_frame=1024):
    """Second token set of the video workload: [frames*tpf, K] viewed as
    [frames, tpf, K] and transposed to [tpf, frames, K] (temporal attention
    groups one spatial position across frames).  A pure row permutation."""
    K = X.shape[-1]
    return (X.reshape(frames, tokens_per_frame, K).transpose(0, 1)
            .reshape(frames * tokens_per_frame, K).contiguous())
