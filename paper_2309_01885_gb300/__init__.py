"""QuantEase layer-wise quantization (arXiv 2309.01885) on one GB300.

The compute path is libqe.so (hand-written sm_103a kernels behind the C ABI of
include/qe.h); ``paper_2309_01885_gb300.qe`` is its Python binding and
``paper_2309_01885_gb300.inputs`` the seeded synthetic workloads.  Build the
library with ``paper_2309_01885_gb300.build.build_lib()``.
"""
__all__ = ["qe", "inputs", "build"]
