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

#ifdef __cplusplus
}
#endif
#endif /* JF_OPS_H */
