"""Host-side models in bench.py (no GPU): the GEMM's per-SM intake ceiling
and the rotate-quant byte accounting."""
import os
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import bench  # noqa: E402


def test_intake_bound_by_hand():
    # one layer, 65536 x 3456 x 1152: 512 x 14 = 7168 tiles of 128 x 256 on
    # 152 SMs -> 48 rounds; a tile moves 384 * 1152 + 65536 bytes at
    # 64 B/clk x 2.07 GHz
    t = 48 * (384 * 1152 + 2 * 128 * 256) / (64 * 2070e6)
    want = 2 * 65536 * 3456 * 1152 / t / 1e12
    got = bench.gemm_intake_bound(65536, [(1152, 3456)], 152, 2070, 64.0)
    assert abs(got - want) < 1e-9 * want


def test_intake_bound_picks_192_wide_tiles_when_they_fit():
    # N = 1152 at 8192 tokens: 6 tiles of 192 per row block, 384 tiles, 3 rounds
    t = 3 * (320 * 1152 + 2 * 128 * 192) / (64 * 2070e6)
    want = 2 * 8192 * 1152 * 1152 / t / 1e12
    got = bench.gemm_intake_bound(8192, [(1152, 1152)], 152, 2070, 64.0)
    assert abs(got - want) < 1e-9 * want


def test_rotate_quant_bytes():
    # 2.5 B per element (16-bit input, packed INT4 codes) + a 4-byte scale a row
    assert bench.rq_algorithmic_bytes(8192, 1152) == 8192 * (2.5 * 1152 + 4)
    # the E4M3 layout writes 1 B a code, E2M3 0.75
    assert bench.rq_layout_bytes(10, 128, 1.0) == 10 * (3.0 * 128 + 4)
    assert bench.rq_layout_bytes(10, 128, 0.75) == 10 * (2.75 * 128 + 4)
