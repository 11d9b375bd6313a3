"""GB300-native LUNA linear attention (arXiv 2512.08061): hand-written CUDA for
sm_103a behind a C ABI (include/luna.h), with a thin Python binding.

Importing the package does not load the CUDA library; `import
paper_2512_08061_gb300.luna` does, and raises if it has not been built.
"""

__all__ = ["build", "luna"]
