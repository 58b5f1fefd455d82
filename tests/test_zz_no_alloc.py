"""The scratch-free fused entry point, clq_fused_linear_noalloc.

It serves callers that cannot allocate device memory where they run the layer
(inference-engine plugin hooks, serving loops that forbid allocation once
started): instead of a caller workspace it uses the library's static device
scratch array.  This file runs last (pytest collects it after the others) and
checks, through the C ABI, that two calls in a row, the second smaller than
the first (so stale codes and counters of the first call sit in the shared
array), give bit for bit the output of clq_fused_linear with an ordinary
workspace (the same kernel and arithmetic), that the result matches the
oracle within the parity tests' output tolerance, and that oversized problems
are refused before any launch while empty ones stay no-ops.
"""
import numpy as np
import pytest
import torch

from paper_2509_24416_gb300 import clq
import oracle
from parity_utils import check_output_frobenius

pytestmark = pytest.mark.gpu
DEV = torch.device("cuda:0")


def _layer(seed, M=300, N=600, K=1152, b=64):
    g = torch.Generator().manual_seed(seed)
    X = (torch.randn(M, K, generator=g) * 3).half()
    X[:, torch.randperm(K, generator=g)[:4]] *= 40
    W = (torch.randn(N, K, generator=g) * 0.02).half()
    bias = (torch.randn(N, generator=g) * 0.01).half()
    perm = torch.randperm(K, generator=g).to(torch.int32)
    layer = clq.PreparedLinear.from_weight(W.to(DEV), perm.to(DEV), b, bias=bias.to(DEV))
    return X.to(DEV), layer, W, perm, bias


def _noalloc(X, layer, Y):
    M, K = X.shape
    N = layer.We.shape[0]
    st = clq.clq_fused_linear_noalloc(
        X.data_ptr(), clq.CLQ_F16, M, K, X.stride(0), layer.perm.data_ptr(), layer.b,
        layer.We.data_ptr(), layer.w_codes, layer.s_w.data_ptr(), layer.bias.data_ptr(),
        N, Y.data_ptr(), torch.cuda.current_stream().cuda_stream)
    return st


def test_noalloc_matches_fused_on_two_calls_in_a_row():
    clq.load()
    for seed, M in ((1, 1000), (2, 300)):
        X, layer, W, perm, bias = _layer(seed, M=M)
        ws = clq.fused_workspace(X.shape[0], X.shape[1], DEV)
        ref = clq.fused_linear(X, layer.perm, layer.b, layer.We, layer.s_w, layer.bias,
                               workspace=ws)
        Y = torch.full_like(ref, float("nan"))
        assert _noalloc(X, layer, Y) == 0
        torch.cuda.synchronize()
        assert clq.device_status() == 0
        assert torch.equal(Y, ref)
    # the second (smaller) call against the oracle, with the oracle's own weights
    Wq_o, s_w_o, _, _ = oracle.prepare_weights(W.float().numpy(), perm.numpy(), 64)
    y64 = oracle.fused_linear(X.float().cpu().numpy(), perm.numpy(), 64, Wq_o, s_w_o,
                              bias.float().numpy())
    check_output_frobenius(Y.float().cpu().numpy().astype(np.float64), y64)


def test_noalloc_empty_problem_is_a_noop_at_any_size():
    # N = 0: nothing to compute, even where M x K is beyond the scratch limit
    P = 1 << 20  # never dereferenced
    st = clq.clq_fused_linear_noalloc(P, clq.CLQ_F16, 65536, 2048, 2048, P, 64, P,
                                      clq.CLQ_CODES_E4M3, P, None, 0, P, None)
    assert st == 0


def test_noalloc_refuses_problems_beyond_the_scratch_limit():
    # 65536 tokens x 2048 channels need 128 MiB of E4M3 codes: too big.
    M, K = 65536, 2048
    assert clq.clq_fused_linear_workspace_size(M, K) > (64 << 20)
    P = 1 << 20  # never dereferenced: the call must return before launching
    st = clq.clq_fused_linear_noalloc(P, clq.CLQ_F16, M, K, K, P, 64, P,
                                      clq.CLQ_CODES_E4M3, P, None, 128, P, None)
    assert st == 8  # CLQ_ERR_SCRATCH_LIMIT
