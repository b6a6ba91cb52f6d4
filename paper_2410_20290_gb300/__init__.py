"""libsr: Speculative Rejection (arXiv 2410.20290) on one GB300 GPU.

The compute path is the CUDA library built from ``csrc/`` (C ABI in include/sr.h);
``binding`` is its ctypes binding.  Build with ``python -m paper_2410_20290_gb300.build``.
"""
