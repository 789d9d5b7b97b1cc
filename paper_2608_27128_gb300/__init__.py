"""GB300 (sm_103a) TwinKV key-redundancy audit and repair pass (arXiv 2608.27128).

The compute lives in libtwinkv.so (C ABI in include/twinkv.h); ``twinkv`` is its
Python binding.  ``synth`` draws the seeded synthetic workloads.
"""
