"""CPU oracle for the CLQ W4A4 OBS linear layer (test infrastructure only).

Only tests, the smoke check and the benchmark's CPU-baseline leg may import
this package; the product path never does.
"""
from .clq_oracle import *  # noqa: F401,F403
from .clq_oracle import QMAX  # noqa: F401
