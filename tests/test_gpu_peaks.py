"""The peak-rate microbenchmarks behind the measured denominators run through
the C ABI, leave no device error, and give rates in a sane order: the
tcgen05 E4M3 MMA above the warp-level e4m3 MMA, which is above the warp-level
s8 MMA, and an HBM read rate between 1 and 20 TB/s."""
import pytest
import torch

from paper_2509_24416_gb300 import clq

pytestmark = pytest.mark.gpu


def test_peaks_run_and_are_ordered():
    clq.load()
    p = clq.measure_peaks(reps=1)
    torch.cuda.synchronize()
    assert clq.device_status() == 0
    assert all(v > 0 for v in p.values()), p
    assert p["tcgen05_e4m3_tflops"] > p["mma_sync_e4m3_tflops"], p
    assert p["mma_sync_e4m3_tflops"] > p["mma_sync_s8_tops"], p
    assert 1000.0 < p["hbm_read_gbs"] < 20000.0, p
