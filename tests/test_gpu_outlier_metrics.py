"""GPU outlier scores under every metric of Sec. 4.4 (absmax, percentile,
top-k mean, range, PAR) against the oracle: bit-identical fp32 scores and
identical swap vectors, for fp16 and bf16 calibration data, token counts
from 1 to the 16384 limit (powers of two and not), spikes and all-zero
channels."""
import numpy as np
import pytest
import torch

import oracle
from paper_2509_24416_gb300 import clq

pytestmark = pytest.mark.gpu
DEV = torch.device("cuda:0")
METRICS = ["absmax", "percentile", "topk_mean", "range", "par"]


def _calib(B, T, K, dtype, seed):
    g = torch.Generator().manual_seed(seed)
    x = torch.randn(B, T, K, generator=g)
    if K > 3:
        x[:, :, 1] *= 30.0
        x[:, :, 2] = 0.0
    if T > 5:
        x[:, 5, 0] += 200.0
    t = x.to({"f16": torch.float16, "bf16": torch.bfloat16}[dtype])
    return t, t.float().numpy()


@pytest.mark.parametrize("metric", METRICS)
@pytest.mark.parametrize("B,T,K,dtype", [(4, 256, 1152, "f16"), (2, 1000, 37, "bf16"),
                                         (1, 1, 5, "f16"), (3, 16384, 8, "bf16"),
                                         (2, 77, 300, "f16")])
def test_scores_match_oracle_bit_for_bit(metric, B, T, K, dtype):
    t, x32 = _calib(B, T, K, dtype, seed=T + K)
    got = clq.outlier_scores(t.to(DEV), metric=metric).cpu().numpy()
    ref = oracle.outlier_scores(x32, metric)
    assert clq.device_status() == 0
    assert np.array_equal(got.view(np.uint32), ref.view(np.uint32)), (got, ref)
    assert np.array_equal(clq.build_permutation(torch.from_numpy(got)).numpy(),
                          oracle.build_permutation(ref))


def test_metric_entry_with_absmax_equals_method_scores():
    t, _ = _calib(3, 300, 260, "bf16", seed=5)
    t = t.to(DEV)
    ref = clq.outlier_scores(t, metric="absmax")
    got = torch.empty_like(ref)
    rc = clq.clq_outlier_scores_metric(t.data_ptr(), 1, 3, 300, 260, 0, got.data_ptr(), None)
    torch.cuda.synchronize()
    assert rc == 0
    assert torch.equal(got.view(torch.int32), ref.view(torch.int32))
