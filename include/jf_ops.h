/*
 * jf_ops.h -- single kernels of the libjf hot path, exposed for kernel-level parity tests.
 *
 * These run one kernel of the forward pass of Jacobi Forcing's Jacobi iteration (arXiv
 * 2512.14681, Sec. 2.1 Eq. 3: one pass over all in-flight rows) on caller-owned device buffers,
 * outside any context. Same conventions as jf.h: plain pointers, the caller owns all memory,
 * work is ordered on `cuda_stream` (NULL = legacy default stream) and the call does not
 * synchronise; arguments are validated on the host before any launch.
 */
#ifndef JF_OPS_H
#define JF_OPS_H

#include <stddef.h>
#include <stdint.h>

#include "jf.h"

#ifdef __cplusplus
extern "C" {
#endif

/* Device workspace bytes jf_op_gemm needs for this shape (split-K partial tiles and tile
 * tickets). k_splits <= 0 selects the split the forward pass uses for this weight shape. */
jf_status jf_op_gemm_workspace_bytes(int N, int K, int M, int k_splits, size_t* out_bytes);

/* Projection Y[m, n] = sum_k X[m, k] * W[n, k] (fp32 accumulate), the weight-streaming GEMM of
 * every projection of the forward pass.
 * dtype JF_BF16: W [N][K] and X [M][K] bf16 (device, 16-byte aligned, K % 8 == 0), tcgen05
 *   tensor cores fed by TMA; JF_F32: W, X fp32, CUDA cores.
 * Y: device fp32 [M][N]. workspace: device, jf_op_gemm_workspace_bytes() bytes, zero-filled
 * before its first use (the kernel leaves its tickets at zero again). err_word: device int that
 * receives a device error code (0 = none); the caller reads it after synchronising. */
jf_status jf_op_gemm(int dtype, const void* W, const void* X, float* Y, int N, int K, int M, int k_splits,
                     void* workspace, size_t workspace_bytes, int* err_word, void* cuda_stream);

/* Size of the fixed device scratch of jf_op_gemm_noalloc (8 MiB). */
#define JF_OP_GEMM_NOALLOC_SCRATCH_BYTES (8u << 20)

/* jf_op_gemm without a workspace, for callers that cannot allocate device memory: code running
 * inside a device-memory allocator's own hooks, or a process whose device memory is entirely
 * reserved by another pool, cannot obtain the workspace jf_op_gemm asks for. (The paper has no
 * counterpart; this is a library facility.)
 * dtype is bf16 only: W [N][K], X [M][K] bf16 (device, 16-byte aligned, K % 8 == 0), Y fp32 [M][N].
 * The split-K scratch is one static device array of JF_OP_GEMM_NOALLOC_SCRATCH_BYTES that every GPU
 * loading libjf holds until the process exits; a shape whose jf_op_gemm_workspace_bytes() exceeds
 * it is refused with JF_ECAPACITY before any launch. The call allocates nothing (no cudaMalloc,
 * no cudaFree, no allocating library routine). Its first call on a device looks up the array's
 * device address (cudaGetSymbolAddress) and sets that device's kernel attributes, so make that
 * first call before any stream capture. Under CUDA's lazy module loading (the default) that first
 * look-up may also be what loads libjf's device code onto the device and reserves the array there:
 * make the first call at start-up, before another pool takes the device memory, or run with
 * CUDA_MODULE_LOADING=EAGER so that the array is reserved when the library is loaded. All calls share the array: calls that may overlap on the GPU (other streams,
 * other threads) race on it and must be serialised by the caller; each call re-zeroes the tickets
 * it uses before its kernel runs. err_word and cuda_stream as in jf_op_gemm. */
jf_status jf_op_gemm_noalloc(const void* W, const void* X, float* Y, int N, int K, int M, int k_splits,
                             int* err_word, void* cuda_stream);

#ifdef __cplusplus
}
#endif
#endif /* JF_OPS_H */
