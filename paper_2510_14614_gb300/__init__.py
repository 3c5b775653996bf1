"""GB300-native (sm_103a) training hot path for GPT / FAL / FAL+ decoder stacks.

The compute lives in the CUDA shared library ``libfal.so`` (C ABI declared in
``include/fal.h``); ``paper_2510_14614_gb300.fal`` is the ctypes binding.
Importing the package does not load the library.
"""
