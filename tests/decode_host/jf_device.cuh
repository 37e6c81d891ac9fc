// Host stand-in for the kernels' device header, used only by the tests to compile the decoding
// state machine (csrc/jf_decode.cu) for the CPU. Every kernel runs as a single thread
// (threadIdx.x = 0, blockDim.x = 1): the block-strided loops then visit every index in order, the
// parts guarded by threadIdx.x == 0 run as written, and barriers have nothing to order.
#pragma once
#include <cstdint>

#include <cuda_runtime.h>

#include "jf_decode.h"

namespace jf_host {
extern uint3 thread_idx, block_idx;
extern dim3 block_dim, grid_dim;
int* dyn_smem();  // the kernel's dynamic shared memory
// Draft-injection hook: a scripted token for (position, iteration) when the test gave a script,
// else the kernel's own rule (passed in).
typedef int (*inject_fn)(const jf::GenCfg&, int, int, int, int, int*);
int scripted_inject(const jf::GenCfg& g, int seq, int x, int P0, int it, int* err, inject_fn rule);
}  // namespace jf_host

#define threadIdx jf_host::thread_idx
#define blockIdx jf_host::block_idx
#define blockDim jf_host::block_dim
#define gridDim jf_host::grid_dim

inline void __syncthreads() {}
// the kernels' optional timeline records are not part of this build
enum TlKernel : unsigned { TL_ACCEPT = 21, TL_COMMIT = 22 };
#define JF_TL_ENTRY() \
  do {                \
  } while (0)
#define JF_TL_WAITED() \
  do {                 \
  } while (0)
#define JF_TL_EXIT(kid) \
  do {                  \
  } while (0)
inline void pdl_wait() {}
inline void pdl_launch_dependents() {}
inline void jf_set_error(int* err, int code) {
  if (err && *err == 0) *err = code;  // first writer wins, as the device's atomicCAS
}
