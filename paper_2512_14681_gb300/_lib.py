"""ctypes binding of libjf (include/jf.h, include/jf_ops.h): argument marshalling only.

PyTorch provides device memory (the context's arena, op buffers) and CUDA streams; every step of
the Jacobi iteration runs in libjf's kernels. There is no CPU fallback: if libjf.so is missing,
load() raises.
"""
from __future__ import annotations

import ctypes as C
import os

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "_build", "libjf.so")

JF_OK, JF_EINVAL, JF_ENOMEM, JF_ECAPACITY, JF_ESTATE, JF_EIO, JF_ECUDA, JF_EDEVICE, JF_ETIMEOUT, JF_EUNSUPPORTED = range(10)
STATUS_NAMES = ["JF_OK", "JF_EINVAL", "JF_ENOMEM", "JF_ECAPACITY", "JF_ESTATE", "JF_EIO", "JF_ECUDA", "JF_EDEVICE",
                "JF_ETIMEOUT", "JF_EUNSUPPORTED"]
JF_F32, JF_BF16 = 0, 1
JF_BLOCK_RA, JF_BLOCK_PSEUDO, JF_BLOCK_CAND = 0, 1, 2
JF_MODE_BLOCK, JF_MODE_WINDOW, JF_MODE_AR = 0, 1, 2
JF_INIT_REPEAT, JF_INIT_INJECT = 0, 1

# every symbol declared in include/jf.h and include/jf_ops.h
EXPORTS = [
    "jf_arena_bytes", "jf_create", "jf_destroy", "jf_last_error", "jf_init_random_weights", "jf_load_weights",
    "jf_save_weights", "jf_get_weights", "jf_prefill", "jf_truncate", "jf_seq_len", "jf_jacobi_step",
    "jf_forward_logits", "jf_generate", "jf_generate_device", "jf_set_profiling", "jf_kernel_time",
    "jf_op_gemm_workspace_bytes", "jf_op_gemm", "jf_op_gemm_noalloc", "jf_tl_enable", "jf_trajectory_noisy_blocks",
    "jf_set_wait_limit", "jf_wait_limit_probe",
]
JF_OP_GEMM_NOALLOC_SCRATCH_BYTES = 8 << 20


class JfError(RuntimeError):
    def __init__(self, status: int, msg: str):
        self.status = status
        name = STATUS_NAMES[status] if 0 <= status < len(STATUS_NAMES) else str(status)
        super().__init__(f"{name}: {msg}")


class ModelConfig(C.Structure):
    _fields_ = [("n_layers", C.c_int), ("d_model", C.c_int), ("n_heads", C.c_int), ("n_kv_heads", C.c_int),
                ("head_dim", C.c_int), ("d_ff", C.c_int), ("vocab", C.c_int), ("rms_eps", C.c_double),
                ("rope_theta", C.c_double), ("dtype", C.c_int), ("qkv_bias", C.c_int), ("tie_embeddings", C.c_int)]


class RuntimeConfig(C.Structure):
    _fields_ = [("max_seqs", C.c_int), ("max_ctx", C.c_int), ("max_rows", C.c_int), ("logits_rows", C.c_int),
                ("device_arena", C.c_void_p), ("arena_bytes", C.c_size_t), ("cuda_stream", C.c_void_p),
                ("page_size", C.c_int), ("max_segments", C.c_int)]


class Block(C.Structure):
    _fields_ = [("kind", C.c_int), ("start_pos", C.c_int), ("len", C.c_int), ("parent", C.c_int)]


class GenParams(C.Structure):
    _fields_ = [("block_size", C.c_int), ("n_blocks", C.c_int), ("spawn_ratio", C.c_double),
                ("pool_size", C.c_int), ("ngram_len", C.c_int), ("cand_per_iter", C.c_int), ("mode", C.c_int),
                ("init", C.c_int), ("inject_p", C.c_float), ("seed", C.c_uint64), ("max_new", C.c_int),
                ("eos_id", C.c_int), ("truth", C.c_void_p), ("truth_len", C.c_int), ("block_sizes", C.c_void_p),
                ("join_iters", C.c_void_p), ("prefill_chunk", C.c_int)]


class GenStats(C.Structure):
    _fields_ = [("iterations", C.c_int), ("accepted", C.POINTER(C.c_int32)), ("rows", C.POINTER(C.c_int32)),
                ("accepted_cap", C.c_int), ("prefill_ms", C.c_double), ("decode_ms", C.c_double),
                ("kernel_launches", C.c_longlong), ("iter_ms", C.POINTER(C.c_float)), ("traj", C.c_void_p),
                ("traj_cap", C.c_int), ("traj_rows", C.c_int), ("traj_iters", C.c_int)]


_lib = None


def load():
    """Load libjf.so; raises if it has not been built (there is no fallback path)."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(LIB_PATH):
        raise RuntimeError(f"libjf.so not built ({LIB_PATH}); run __graft_entry__.build()")
    L = C.CDLL(LIB_PATH)
    vp, i32, st, P = C.c_void_p, C.c_int, C.c_int, C.POINTER
    L.jf_arena_bytes.argtypes = [P(ModelConfig), P(RuntimeConfig), P(C.c_size_t)]
    L.jf_create.argtypes = [P(ModelConfig), P(RuntimeConfig), P(vp)]
    L.jf_destroy.argtypes = [vp]
    L.jf_destroy.restype = None
    L.jf_last_error.argtypes = [vp]
    L.jf_last_error.restype = C.c_char_p
    L.jf_init_random_weights.argtypes = [vp, C.c_uint64, C.c_double]
    L.jf_load_weights.argtypes = [vp, C.c_char_p]
    L.jf_save_weights.argtypes = [vp, C.c_char_p]
    L.jf_get_weights.argtypes = [vp, i32, C.c_longlong, C.c_longlong, P(C.c_float)]
    L.jf_prefill.argtypes = [vp, i32, P(C.c_int32), i32, P(C.c_int32)]
    L.jf_truncate.argtypes = [vp, i32, i32]
    L.jf_seq_len.argtypes = [vp, i32, P(C.c_int)]
    L.jf_jacobi_step.argtypes = [vp, i32, i32, P(Block), P(C.c_int32), P(C.c_int32), P(C.c_int32), P(C.c_int32),
                                 P(C.c_int32), P(C.c_float)]
    L.jf_forward_logits.argtypes = [vp, i32, i32, P(C.c_int32), P(C.c_float), P(C.c_float), P(C.c_int32)]
    L.jf_generate.argtypes = [vp, i32, P(P(C.c_int32)), P(C.c_int32), P(GenParams), P(C.c_int32), P(GenStats)]
    L.jf_generate_device.argtypes = [vp, i32, vp, P(C.c_int32), P(GenParams), vp, P(GenStats)]
    L.jf_set_profiling.argtypes = [vp, i32]
    L.jf_kernel_time.argtypes = [vp, i32, P(C.c_double), P(C.c_longlong)]
    L.jf_op_gemm_workspace_bytes.argtypes = [i32, i32, i32, i32, P(C.c_size_t)]
    L.jf_op_gemm.argtypes = [i32, vp, vp, vp, i32, i32, i32, i32, vp, C.c_size_t, vp, vp]
    L.jf_op_gemm_noalloc.argtypes = [vp, vp, vp, i32, i32, i32, i32, vp, vp]
    L.jf_tl_enable.argtypes = [vp, vp]
    L.jf_trajectory_noisy_blocks.argtypes = [vp, i32, i32, i32, vp, i32, i32, i32, i32, vp, vp, vp]
    L.jf_set_wait_limit.argtypes = [vp, C.c_uint64]
    L.jf_wait_limit_probe.argtypes = [vp, P(C.c_uint64)]
    for name in EXPORTS:
        f = getattr(L, name)
        if name not in ("jf_destroy", "jf_last_error"):
            f.restype = st
    _lib = L
    return L
