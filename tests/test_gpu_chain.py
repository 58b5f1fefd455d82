"""Layers chained on one stream: each layer's input is the output that the
previous layer's GEMM wrote just before.  The library's kernels launch with
programmatic dependent launch, so a rotate-quant grid may start while the
GEMM before it drains; it prefetches its first tiles into L2 meanwhile and
reads its input only after the wait.  The chained outputs must equal the same
calls with a device synchronization between layers, bit for bit, with every
intermediate buffer filled with NaN on the stream first (an input read too
early would carry the NaN through), for each rotate-quant loop: the wide loop
(b = 64), the paired loop (b = 128), the general loop (8-bit activations, and
asymmetric 4-bit codes at b = 32), and the fused kernel; and weights
prepared right after torch kernels computed their swap vector."""
import pytest
import torch

from paper_2509_24416_gb300 import clq

pytestmark = pytest.mark.gpu
DEV = torch.device("cuda:0")
M = 4096
WIDTHS = (1152, 1152, 2304, 1152)  # K of the first layer, then each layer's N


def _layers(seed, b, a_bits=4, w_bits=4, dtype=torch.float16):
    g = torch.Generator().manual_seed(seed)
    out = []
    for K, N in zip(WIDTHS[:-1], WIDTHS[1:]):
        W = (torch.randn(N, K, generator=g) * (1.0 / K ** 0.5)).to(dtype).to(DEV)
        bias = (torch.randn(N, generator=g) * 0.01).to(dtype).to(DEV)
        perm = torch.randperm(K, generator=g).to(torch.int32).to(DEV)
        out.append(clq.PreparedLinear.from_weight(W, perm, b, bias=bias, a_bits=a_bits,
                                                  w_bits=w_bits))
    return out


def _check_chain(run_layer, x0, reps=3):
    ref = []
    x = x0
    for i in range(len(WIDTHS) - 1):
        y = torch.empty((M, WIDTHS[i + 1]), dtype=x0.dtype, device=DEV)
        run_layer(i, x, y)
        torch.cuda.synchronize()
        ref.append(y)
        x = y
    assert all(bool(torch.isfinite(r).all()) for r in ref)
    ys = [torch.empty_like(r) for r in ref]
    for _ in range(reps):
        for y in ys:
            y.fill_(float("nan"))
        x = x0
        for i, y in enumerate(ys):
            run_layer(i, x, y)
            x = y
        torch.cuda.synchronize()
        assert clq.device_status() == 0
        for y, r in zip(ys, ref):
            assert torch.equal(y.view(torch.int16), r.view(torch.int16))


def _x0(seed, dtype=torch.float16):
    g = torch.Generator().manual_seed(seed)
    return (torch.randn(M, WIDTHS[0], generator=g) * 3).to(dtype).to(DEV)


@pytest.mark.parametrize("b,a_bits,fused,dtype", [(64, 4, False, torch.float16),
                                                  (128, 4, False, torch.float16),
                                                  (64, 8, False, torch.float16),
                                                  (64, 4, True, torch.float16),
                                                  (64, 4, False, torch.bfloat16),
                                                  (128, 4, False, torch.bfloat16)])
def test_chained_layers_equal_synchronized(b, a_bits, fused, dtype):
    layers = _layers(11, b, a_bits=a_bits, dtype=dtype)
    ws = [clq.fused_workspace(M, K, DEV) if fused else None for K in WIDTHS[:-1]]

    def run_layer(i, x, y):
        layers[i](x, fused=fused, workspace=ws[i], Y=y)

    _check_chain(run_layer, _x0(12, dtype))


def test_chained_asymmetric_layers_equal_synchronized():
    b = 32
    layers = _layers(13, b)
    wsums = [clq.weight_code_sums(lay.We, K)
             for lay, K in zip(layers, WIDTHS[:-1])]

    def run_layer(i, x, y):
        lay = layers[i]
        K = WIDTHS[i]
        Xq, delta, lo = clq.rotate_quant_act_asym(x, lay.perm, b)
        clq.linear_asym(Xq, delta, lo, lay.We, lay.s_w, wsums[i], b, K, bias=lay.bias, Y=y)

    _check_chain(run_layer, _x0(14))


def test_weights_prepared_right_after_a_device_swap_vector():
    """Weight preparation launches without programmatic overlap, so a swap
    vector that torch kernels compute on the device just before it is read
    complete: the prepared codes and scales equal those from the same swap
    vector copied in after a synchronization."""
    K, N, b = 1152, 640, 64
    g = torch.Generator().manual_seed(21)
    W = (torch.randn(N, K, generator=g) * 0.02).half().to(DEV)
    scores = torch.rand(K, generator=g).to(DEV)
    torch.cuda.synchronize()
    for _ in range(3):
        perm_dev = torch.argsort(scores, descending=True).to(torch.int32)  # device kernels
        lay = clq.PreparedLinear.from_weight(W, perm_dev, b)
        torch.cuda.synchronize()
        ref = clq.PreparedLinear.from_weight(W, perm_dev.cpu().to(DEV), b)
        torch.cuda.synchronize()
        assert clq.device_status() == 0
        assert torch.equal(lay.We, ref.We) and torch.equal(lay.s_w, ref.s_w)
        scores = scores.roll(1)
