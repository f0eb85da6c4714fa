"""GB300 (sm_103a) dense GEMM C = A.B: int8 x int8 -> exact int32, and
bf16 x bf16 -> fp32 accumulation -> round-to-nearest-even bf16.

The compute lives in a C-ABI shared library of hand-written CUDA kernels
(``csrc/``, declared in ``include/gb300_gemm.h``); ``gemm`` is its thin ctypes
binding with the same names.  ``workloads`` holds the seeded synthetic input
generators and holds none of the GEMM arithmetic.

Importing the package loads nothing; the binding loads the library on first
use and raises if it has not been built.
"""

__all__ = ["gemm", "workloads"]
