"""GB300 (sm_103a) N-MDLM spiking block-denoise library.

``api`` holds the PyTorch-facing wrappers of the C ABI in include/nmdlm.h; ``synth``
the seeded synthetic inputs.  Importing the package loads nothing; the CUDA library is
loaded (and built in-tree if needed) by the first ``api.Context``.
"""
__all__ = ["api", "synth", "build"]
