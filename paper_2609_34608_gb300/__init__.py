"""GB300-native (sm_103a) WAMachine hot path: a C-ABI CUDA library and its Python binding.

Importing the package is cheap; the shared library is loaded by ``paper_2609_34608_gb300.wam``
on first use and raises if it has not been built.
"""
__all__ = ["inputs"]
