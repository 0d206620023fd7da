"""GB300-native schedule-driven cached denoising (EVO hot path).

The compute path lives in ``csrc/`` (CUDA for sm_103a behind a C ABI declared
in ``include/evo.h``); ``binding`` loads that library with ctypes.  Importing
this package does not load the library; ``binding.load()`` does, and raises if
it is missing.
"""
