"""GB300-native dual-sparse batch-1 spMspV (DuoGPT, arXiv 2506.20194).

The compute path lives in ``libduo.so`` (hand-written CUDA for sm_103a behind
a C ABI, ``include/duo.h``); :mod:`paper_2506_20194_gb300.duo` is a thin
ctypes binding with the same entry-point names.  :mod:`.synth` draws seeded
synthetic inputs.  Importing this package does not load the library.
"""
