"""Permutation-group Allreduce (Kolmakov & Zhang, arXiv 2004.09362) on one GB300.

The C-ABI library libgar.so (include/gar.h) holds the schedule builder and the CUDA
kernels; ``paper_2004_09362_gb300.gar`` is its Python binding and
``paper_2004_09362_gb300.build`` compiles the library.  Import the binding explicitly:
``from paper_2004_09362_gb300 import gar``.
"""
