"""clq.HostPipeline: pinned host inputs -> host outputs through the public
API with copies and kernels on three streams.  The outputs equal direct
PreparedLinear calls bit for bit, on two passes in a row (the second pass
reuses every device buffer while the first may still be in flight), for the
separate and the fused path."""
import pytest
import torch

from paper_2509_24416_gb300 import clq

pytestmark = pytest.mark.gpu
DEV = torch.device("cuda:0")


def _layers(seed, shapes, b=64, bits=(4, 4)):
    g = torch.Generator().manual_seed(seed)
    out = []
    for (M, K, N) in shapes:
        W = (torch.randn(N, K, generator=g) * 0.02).half().to(DEV)
        bias = (torch.randn(N, generator=g) * 0.01).half().to(DEV)
        perm = torch.randperm(K, generator=g).to(torch.int32).to(DEV)
        out.append((clq.PreparedLinear.from_weight(W, perm, b, bias=bias, a_bits=bits[0],
                                                   w_bits=bits[1]), M, K, N))
    return out


@pytest.mark.parametrize("fused", [False, True])
def test_host_pipeline_matches_direct_calls(fused):
    shapes = [(300, 1152, 640), (129, 1152, 1152), (64, 4608, 256)]
    layers = _layers(3, shapes)
    g = torch.Generator().manual_seed(4)
    passes = []
    for p in range(2):
        xh = [(torch.randn(M, K, generator=g) * 3).half().pin_memory() for (_, M, K, _) in layers]
        yh = [torch.empty((M, N), dtype=torch.float16).pin_memory() for (_, M, _, N) in layers]
        passes.append((xh, yh))
    pipe = clq.HostPipeline(layers, torch.float16, DEV, fused=fused)
    for xh, yh in passes:
        pipe.run(xh, yh)
    pipe.join()
    torch.cuda.synchronize()
    assert clq.device_status() == 0
    for xh, yh in passes:
        for (lay, M, K, N), x, y in zip(layers, xh, yh):
            ref = lay(x.to(DEV), fused=fused).cpu()
            assert torch.equal(y.view(torch.int16), ref.view(torch.int16))


@pytest.mark.parametrize("bits", [(8, 4), (8, 8)])
def test_host_pipeline_8bit_layers(bits):
    """8-bit activation codes need twice the code buffer; the pipeline sizes
    it from each layer's bit setting."""
    shapes = [(200, 1152, 384), (96, 4608, 512)]
    layers = _layers(5, shapes, bits=bits)
    g = torch.Generator().manual_seed(6)
    xh = [(torch.randn(M, K, generator=g) * 3).half().pin_memory() for (_, M, K, _) in layers]
    yh = [torch.empty((M, N), dtype=torch.float16).pin_memory() for (_, M, _, N) in layers]
    pipe = clq.HostPipeline(layers, torch.float16, DEV)
    pipe.run(xh, yh)
    pipe.run(xh, yh)
    pipe.join()
    torch.cuda.synchronize()
    assert clq.device_status() == 0
    for (lay, M, K, N), x, y in zip(layers, xh, yh):
        ref = lay(x.to(DEV)).cpu()
        assert torch.equal(y.view(torch.int16), ref.view(torch.int16))
