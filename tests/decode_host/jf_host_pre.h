// Force-included first when the decoding kernels are compiled for the CPU (tests only): the CUDA
// runtime header for its host types, then the CUDA qualifiers as plain C++.
#pragma once
#include <cuda_runtime.h>
#undef __device__
#undef __global__
#undef __host__
#undef __shared__
#undef __forceinline__
#define __device__
#define __global__
#define __host__
#define __shared__ static
#define __forceinline__ inline
