"""GB300-native Parser Stack Classification (PSC) for grammar-constrained decoding.

The library (``libpsc_gb300.so``, C ABI in ``include/psc.h``) compiles a grammar and
a vocabulary into a stack classifier and precomputed masks, and runs the per-step
mask computation, masking and sampling in CUDA kernels for sm_103a.  ``psc`` is
its thin Python binding.
"""
