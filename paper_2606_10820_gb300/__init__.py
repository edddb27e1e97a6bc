"""GB300 (sm_103a) implementation of K-Forcing's joint next-k-token decode step.

The compute lives in ``libkforcing.so`` (CUDA kernels behind the C ABI of
include/kforcing.h); ``kforcing`` is its Python binding and ``build`` compiles
it.  Importing the package loads nothing; the binding raises if the library
has not been built.
"""
