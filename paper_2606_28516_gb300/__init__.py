"""GB300 (sm_103a) CLEAR-MoE FFN layer: hand-written CUDA behind a small C ABI.

The compute lives in libclearmoe.so (paper_2606_28516_gb300/csrc, declared in include/clearmoe.h);
`clearmoe` is the ctypes binding with the same names. Importing the package loads nothing; the
binding fails loudly if the library has not been built (paper_2606_28516_gb300.build.build()).
"""
