"""GB300-native integer-only quantized convolution of AQD (arXiv 2007.06919).

``aqd`` is the ctypes binding of libaqd.so (C ABI in include/aqd.h); ``synth`` draws the
seeded synthetic workloads; ``build`` compiles the CUDA sources for sm_103a in-tree.
"""
