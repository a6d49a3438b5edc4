"""GB300-native action-expert tick (fast system of an asynchronous fast-slow
driving agent): a C-ABI CUDA library plus a thin ctypes binding.

Importing the package loads nothing; ``paper_2607_15621_gb300.fsx`` loads the
compiled library and fails loudly when it is missing.
"""
__all__ = ["fsx", "synth", "build"]
