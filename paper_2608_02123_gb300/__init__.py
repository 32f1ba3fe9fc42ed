"""PCTree drafting round for NVIDIA GB300 (sm_103a).

The compute path is the CUDA library built from ``csrc/`` (C ABI in
``include/pctree.h``); ``paper_2608_02123_gb300.pctree`` is its Python
binding.  Importing the binding fails if the library has not been built.
"""
__all__ = ["pctree"]
