"""GB300-native stale-synchronous parameter table for MF-SGD (arXiv 1410.8043).

The CUDA library (csrc/, C-ABI in include/esspt.h) is built in-tree by
`paper_1410_8043_gb300.build.build()`; `paper_1410_8043_gb300.esspt` is its
Python binding.  Importing the package does not load the library.
"""

__all__ = ["build", "esspt"]
