"""The peak-rate microbenchmarks behind the measured denominators run through
the C ABI, leave no device error, and give rates in a sane order: the
tcgen05 E4M3 MMA above the warp-level e4m3 MMA, which is above the warp-level
s8 MMA, and an HBM read rate between 1 and 20 TB/s.  The rotate-quant memory
floor writes the high byte of every input value and a 4-byte value per row,
and reports the kernel's algorithmic bytes."""
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


def test_rq_stream_floor_moves_the_bytes():
    import ctypes
    clq.load()
    dev = torch.device("cuda:0")
    for M, K in ((1000, 1152), (37, 4608), (8192, 1152)):
        X = torch.randint(-32768, 32767, (M, K), dtype=torch.int16, device=dev)
        Q = torch.zeros((M, K), dtype=torch.uint8, device=dev)
        S = torch.zeros(M, dtype=torch.float32, device=dev)
        ops = ctypes.c_int64(0)
        st = clq.clq_peak_rq_stream(X.data_ptr(), M, K, Q.data_ptr(), S.data_ptr(),
                                    ctypes.byref(ops), torch.cuda.current_stream().cuda_stream)
        assert st == 0, st
        torch.cuda.synchronize()
        assert clq.device_status() == 0
        assert ops.value == M * (5 * K // 2 + 4)
        hi = (X.view(torch.uint8).view(M, K, 2)[:, :, 1])
        assert torch.equal(Q, hi)
        assert bool((S == 1.0).all())
