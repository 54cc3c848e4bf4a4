"""GB300-native rotated-hypercube mixing layer (arXiv 2609.18145).

The compute path is libhcw.so (CUDA for sm_103a) behind the C ABI of
include/hcw.h; ``paper_2609_18145_gb300.hcw`` is its Python binding and
``paper_2609_18145_gb300.synth`` the seeded synthetic inputs.
"""
from ._build import LIB, build  # noqa: F401
