"""NeuRoute batched query path for GB300 (sm_103a).

The compute path is the C-ABI library ``libneuroute.so`` (hand-written CUDA
kernels, declared in ``include/neuroute.h``); ``neuroute`` is its ctypes
binding. The index file is produced by ``builder`` (a host routine run once,
off the query path).
"""
