"""GPU parity for the per-layer clip search (Sec. 3.4, Eq. 3, the layer as
its own target): the clip table and the chosen bounds against the oracle's,
each grid point's squared error against the oracle's fp64 error, and the
chosen percentile near-optimal under the oracle's objective.

Tolerance for the errors e = ||Y - Y^||_F^2: the GPU's Y^ is rounded to the
output format (half-ulp u per element, so ||dY^|| <= u ||Y^||) and may hold
rare off-by-one activation codes at rounding ties; then
|e_gpu - e| <= 2 sqrt(e) (1.5 u ||Y^||) + (1.5 u ||Y^||)^2 + 1e-3 e.
Clip bounds come from the GPU's rotated weights (1e-5 of the row's maximum,
as for the rotation itself).
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2509_24416_gb300 import clq, synth

pytestmark = pytest.mark.gpu
DEV = torch.device("cuda:0")
TD = {"f16": torch.float16, "bf16": torch.bfloat16}


@pytest.fixture(scope="module", autouse=True)
def _lib():
    clq.load()
    yield
    assert clq.device_status() == 0


def _run(W32, X32, bias32, perm, b, dtype, grid):
    td = TD[dtype]
    W = torch.from_numpy(W32).to(td)
    X = torch.from_numpy(X32).to(td)
    w32 = W.float().numpy()
    x32 = X.float().numpy()
    bias_t = None if bias32 is None else torch.from_numpy(bias32).to(td)
    b32 = None if bias_t is None else bias_t.float().numpy()
    y64 = oracle.linear_fp64(x32, w32, b32)
    g32 = np.asarray(grid, np.float32)
    clip, errors, best = clq.clip_search(W.to(DEV), torch.from_numpy(perm).to(DEV), b, X.to(DEV),
                                         torch.from_numpy(y64.astype(np.float32)).to(DEV),
                                         None if bias_t is None else bias_t.to(DEV),
                                         grid=tuple(float(v) for v in g32))
    torch.cuda.synchronize()
    oe, obest, oclip, _ = oracle.clip_search(x32, w32, perm, b, b32, g32.astype(np.float64))
    u = 2.0 ** -11 if dtype == "f16" else 2.0 ** -8
    e = errors.numpy()
    # ||Y^|| from the oracle's best point is representative of every point
    yh_norm = np.linalg.norm(y64) * 1.5
    tol = 2 * np.sqrt(oe) * 1.5 * u * yh_norm + (1.5 * u * yh_norm) ** 2 + 1e-3 * oe
    assert np.all(np.abs(e - oe) <= tol), (e, oe, tol)
    assert oe[best] <= oe[obest] + tol[best] + tol[obest]
    K = W32.shape[1]
    w_rot = oracle.rotate(w32, perm, b)
    table = oracle.clip_table(w_rot, oracle.clip_rank(float(g32[best]), K) + 1)
    rowmax = np.max(np.abs(w_rot), axis=1)
    assert np.all(np.abs(clip.cpu().numpy() - table[:, -1]) <= 1e-5 * rowmax)
    return e, best, oe, obest


@pytest.mark.parametrize("dtype", ["f16", "bf16"])
def test_clip_search_clips_a_harmless_outlier(dtype):
    rng = np.random.default_rng(71)
    K, N, M = 128, 64, 128
    W = rng.standard_normal((N, K)).astype(np.float32)
    X = rng.standard_normal((M, K)).astype(np.float32)
    W[:, 9] = 40.0
    X[:, 9] = 0.0
    perm = np.arange(K, dtype=np.int32)
    grid = [0.0, 0.0125, 0.025, 0.0375, 0.05]
    e, best, oe, obest = _run(W, X, None, perm, 1, dtype, grid)
    assert best >= 1 and e[0] > 10 * e[best]


@pytest.mark.parametrize("li", [0, 3])
def test_clip_search_on_a_pixart_layer(li):
    cfg = dict(synth.WORKLOADS["pixart_1024"], M=256)
    d = synth.layer_inputs(cfg, li)
    perm = oracle.build_permutation(oracle.outlier_scores(d["calib"]))
    _run(d["W32"], d["X32"], d["bias32"], perm, d["b"], d["dtype"], clq.CLIP_GRID)


def test_clip_search_grid_of_one_is_unclipped():
    rng = np.random.default_rng(72)
    K, N, M = 256, 40, 64
    W = (rng.standard_normal((N, K)) * 0.05).astype(np.float32)
    X = rng.standard_normal((M, K)).astype(np.float32)
    perm = rng.permutation(K).astype(np.int32)
    e, best, _, _ = _run(W, X, None, perm, 64, "f16", [0.0])
    assert best == 0 and e.shape == (1,)


@pytest.mark.parametrize("metric", ["absmax", "topk_mean"])
def test_prepared_linear_calibrate_runs_the_offline_steps(metric):
    """PreparedLinear.calibrate = outlier scores under the metric, swap
    vector, clip search on the calibration tokens, prepared weights, each
    step equal to its own call."""
    cfg = dict(synth.WORKLOADS["pixart_1024"], M=256)
    d = synth.layer_inputs(cfg, 0)
    b = d["b"]
    calib = torch.from_numpy(d["calib"]).to(TD[d["dtype"]]).to(DEV)
    W, bias = d["W"].to(DEV), d["bias"].to(DEV)
    layer, info = clq.PreparedLinear.calibrate(W, calib, b, bias, metric=metric,
                                               clip_grid=clq.CLIP_GRID)
    scores = clq.outlier_scores(calib, metric=metric)
    perm = clq.build_permutation(scores)
    assert torch.equal(info["perm"].cpu(), perm)
    K = W.shape[1]
    Xcal = calib.reshape(-1, K).contiguous()
    # the target calibrate() uses: fp64 product rounded once to fp32
    Yref = (Xcal.double() @ W.double().t() + bias.double()[None, :]).float()
    clip, errors, best = clq.clip_search(W, perm.to(DEV), b, Xcal, Yref, bias)
    assert best == info["best"] and torch.equal(clip, info["clip"])
    ref = clq.PreparedLinear.from_weight(W, perm.to(DEV), b, bias=bias, clip=clip)
    X = d["X"].to(DEV)
    torch.cuda.synchronize()
    assert torch.equal(layer(X), ref(X))
    # the oracle's permutation from the same calibration batch
    o = oracle.build_permutation(oracle.outlier_scores(d["calib"], metric))
    assert np.array_equal(perm.numpy(), o)
