"""GB300-native Jacobi-decoding hot path of Jacobi Forcing (arXiv 2512.14681).

libjf.so (CUDA kernels for sm_103a + host runtime) behind the C ABI of include/jf.h; this package
holds its build script, a ctypes binding (_lib, jacobi) and the seeded input generators (inputs).
"""
