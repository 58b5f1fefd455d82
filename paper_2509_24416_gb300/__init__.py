"""GB300 (sm_103a) inference path of CLQ's W4A4 OBS linear layer
(arxiv 2509.24416): rotate-quantize and packed INT4 GEMM kernels behind a
C ABI (include/clq.h), with a ctypes binding in ``clq``.

Importing the package does not load the CUDA library; the first call into
``clq`` does, and raises if libclq.so has not been built.
"""
__all__ = ["clq", "synth", "build"]
