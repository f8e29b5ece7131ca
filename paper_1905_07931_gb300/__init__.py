"""GB300-native CSR-weight training step (Lee & Lee, arXiv 1905.07931).

The compute path is the CUDA library built from ``csrc/`` (``libcsrtrain.so``),
reached through the ctypes binding in ``csrtrain``. Importing this package does
not load the library; ``csrtrain.lib()`` does, and raises if it is missing.
"""

__all__ = ["csrtrain", "synth", "train"]
