"""Python face of libjf: a Context owning a device arena (PyTorch memory) and a CUDA stream.

Every method marshals arguments and calls one C entry point of include/jf.h; the Jacobi
iteration itself (forward pass, greedy argmax, acceptance, KV commit, draft bookkeeping) runs in
libjf's CUDA kernels.
"""
from __future__ import annotations

import ctypes as C
from dataclasses import dataclass

import numpy as np

from . import _lib as J
from .inputs import ModelShape


def _check(lib, ctx, status: int):
    if status != J.JF_OK:
        msg = lib.jf_last_error(ctx).decode() if ctx else ""
        raise J.JfError(status, msg)


def _i32p(a):
    return a.ctypes.data_as(C.POINTER(C.c_int32))


def _f32p(a):
    return a.ctypes.data_as(C.POINTER(C.c_float))


@dataclass
class Gen:
    """Generation parameters (see jf_gen_params in include/jf.h)."""
    block_size: int = 8
    n_blocks: int = 1
    spawn_ratio: float = 0.0
    pool_size: int = 0
    ngram_len: int = 0
    cand_per_iter: int = 0
    mode: str = "block"
    init: str = "repeat"
    inject_p: float = 0.0
    seed: int = 0
    max_new: int = 64
    eos_id: int = -1
    block_sizes: tuple | None = None   # per-sequence block sizes (block_size = the largest)
    join_iters: tuple | None = None    # per-sequence join iteration (0 = prefilled first)
    prefill_chunk: int = 0             # rows of one in-iteration prefill chunk (0 = 64)

    def c_struct(self, truth_ptr=None, truth_len=0) -> J.GenParams:
        mode = {"block": J.JF_MODE_BLOCK, "window": J.JF_MODE_WINDOW, "ar": J.JF_MODE_AR}[self.mode]
        init = {"repeat": J.JF_INIT_REPEAT, "inject": J.JF_INIT_INJECT}[self.init]
        gp = J.GenParams(self.block_size, self.n_blocks, self.spawn_ratio, self.pool_size, self.ngram_len,
                         self.cand_per_iter, mode, init, self.inject_p, self.seed, self.max_new, self.eos_id,
                         truth_ptr, truth_len)
        # the per-sequence arrays live as long as the returned structure
        gp._keep = []
        for name in ("block_sizes", "join_iters"):
            v = getattr(self, name)
            if v is not None:
                a = np.ascontiguousarray(v, dtype=np.int32)
                gp._keep.append(a)
                setattr(gp, name, a.ctypes.data)
        gp.prefill_chunk = self.prefill_chunk
        return gp


@dataclass
class GenOut:
    tokens: np.ndarray      # [n_seqs, max_new]
    counts: np.ndarray      # [iterations, n_seqs] tokens committed per iteration (-1 = inactive)
    rows: np.ndarray        # [iterations] in-flight rows per iteration
    iterations: int
    prefill_ms: float
    decode_ms: float
    kernel_launches: int = 0
    iter_ms: np.ndarray | None = None  # [iterations] device time of each iteration's graph replay
    traj_iters: int = 0                # iterations recorded into the trajectory buffer


def trajectory_records(buf, n_iters: int, traj_rows: int):
    """Split a trajectory buffer written by jf_generate (see jf_gen_stats in include/jf.h) into one
    dict per recorded iteration: M, it, and per row seq, kind, pos, token, pred (numpy int32)."""
    a = buf.cpu().numpy() if hasattr(buf, "cpu") else np.asarray(buf)
    a = a.reshape(-1)[: n_iters * (2 + 5 * traj_rows)].reshape(n_iters, 2 + 5 * traj_rows)
    out = []
    for rec in a:
        M = int(rec[0])
        f = [rec[2 + j * traj_rows: 2 + j * traj_rows + M] for j in range(5)]
        out.append(dict(M=M, it=int(rec[1]), seq=f[0], kind=f[1], pos=f[2], token=f[3], pred=f[4]))
    return out


def model_config(shape: ModelShape) -> J.ModelConfig:
    return J.ModelConfig(shape.n_layers, shape.d_model, shape.n_heads, shape.n_kv_heads, shape.head_dim,
                         shape.d_ff, shape.vocab, shape.rms_eps, shape.rope_theta,
                         J.JF_BF16 if shape.bf16 else J.JF_F32, int(shape.qkv_bias), int(shape.tie_embeddings))


class Context:
    """A libjf context on the current CUDA device."""

    def __init__(self, shape: ModelShape, max_seqs: int = 1, max_ctx: int = 2048, max_rows: int = 64,
                 logits_rows: int = 0, stream=None, max_segments: int = 0):
        import torch

        self.lib = J.load()
        self.shape = shape
        self.mc = model_config(shape)
        self.torch = torch
        self.stream = stream if stream is not None else torch.cuda.Stream()
        rc = J.RuntimeConfig(max_seqs, max_ctx, max_rows, logits_rows, None, 0, self.stream.cuda_stream, 16,
                             max_segments)
        nbytes = C.c_size_t()
        _check(self.lib, None, self.lib.jf_arena_bytes(C.byref(self.mc), C.byref(rc), C.byref(nbytes)))
        self.arena = torch.empty(nbytes.value, dtype=torch.uint8, device="cuda")
        rc.device_arena = self.arena.data_ptr()
        rc.arena_bytes = nbytes.value
        self.rc = rc
        h = C.c_void_p()
        torch.cuda.synchronize()
        _check(self.lib, None, self.lib.jf_create(C.byref(self.mc), C.byref(rc), C.byref(h)))
        self.h = h
        self.max_rows = max_rows
        self.max_ctx = max_ctx

    def close(self):
        if getattr(self, "h", None):
            self.lib.jf_destroy(self.h)
            self.h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def _c(self, status):
        _check(self.lib, self.h, status)

    # -- weights -----------------------------------------------------------------------
    def init_random_weights(self, seed: int = 0, std: float = 0.02):
        self._c(self.lib.jf_init_random_weights(self.h, seed, std))

    def save_weights(self, path: str):
        self._c(self.lib.jf_save_weights(self.h, path.encode()))

    def load_weights(self, path: str):
        self._c(self.lib.jf_load_weights(self.h, path.encode()))

    def get_weights(self, tensor_id: int, start: int, count: int) -> np.ndarray:
        out = np.empty(count, dtype=np.float32)
        self._c(self.lib.jf_get_weights(self.h, tensor_id, start, count,
                                        out.ctypes.data_as(C.POINTER(C.c_float))))
        return out

    # -- sequences ---------------------------------------------------------------------
    def prefill(self, seq: int, prompt) -> int:
        p = np.ascontiguousarray(prompt, dtype=np.int32)
        nt = C.c_int32()
        self._c(self.lib.jf_prefill(self.h, seq, _i32p(p), p.size, C.byref(nt)))
        return int(nt.value)

    def truncate(self, seq: int, length: int):
        self._c(self.lib.jf_truncate(self.h, seq, length))

    def seq_len(self, seq: int) -> int:
        v = C.c_int()
        self._c(self.lib.jf_seq_len(self.h, seq, C.byref(v)))
        return int(v.value)

    def jacobi_step(self, seq: int, blocks, draft):
        """blocks: list of (kind, start_pos, len, parent). Returns dict of outputs."""
        bl = (J.Block * len(blocks))(*[J.Block(*b) for b in blocks])
        d = np.ascontiguousarray(draft, dtype=np.int32)
        counts = np.zeros(len(blocks), dtype=np.int32)
        committed = np.zeros(max(b[2] for b in blocks), dtype=np.int32)
        n_comm = C.c_int32()
        pred = np.zeros(d.size, dtype=np.int32)
        top2 = np.zeros((d.size, 2), dtype=np.float32)
        self._c(self.lib.jf_jacobi_step(self.h, seq, len(blocks), bl, _i32p(d), _i32p(counts), _i32p(committed),
                                        C.byref(n_comm), _i32p(pred), top2.ctypes.data_as(C.POINTER(C.c_float))))
        return dict(counts=counts, committed=committed[: n_comm.value], predictions=pred, top2=top2)

    def forward_logits(self, seq: int, tokens, want_logits=True, want_hidden=True):
        t = np.ascontiguousarray(tokens, dtype=np.int32)
        n = t.size
        logits = np.empty((n, self.shape.vocab), dtype=np.float32) if want_logits else None
        hidden = np.empty((n, self.shape.d_model), dtype=np.float32) if want_hidden else None
        am = np.empty(n, dtype=np.int32)
        fp = C.POINTER(C.c_float)
        self._c(self.lib.jf_forward_logits(self.h, seq, n, _i32p(t),
                                           logits.ctypes.data_as(fp) if logits is not None else None,
                                           hidden.ctypes.data_as(fp) if hidden is not None else None, _i32p(am)))
        return logits, hidden, am

    # -- generation --------------------------------------------------------------------
    def generate(self, prompts, gen: Gen, truth=None, log_cap: int = 4096, traj=None, traj_rows: int = 0) -> GenOut:
        """Host buffers in and out (jf_generate). traj: optional device int32 tensor of
        cap * (2 + 5 * traj_rows) elements that receives the Jacobi trajectory records."""
        ps = [np.ascontiguousarray(p, dtype=np.int32) for p in prompts]
        n = len(ps)
        arr = (C.POINTER(C.c_int32) * n)(*[_i32p(p) for p in ps])
        lens = np.array([p.size for p in ps], dtype=np.int32)
        tr = None
        tlen = 0
        if truth is not None:
            tr = np.ascontiguousarray(truth, dtype=np.int32)
            tlen = tr.shape[-1]
        gp = gen.c_struct(tr.ctypes.data if tr is not None else None, tlen)
        out = np.empty((n, gen.max_new), dtype=np.int32)
        acc = np.full((log_cap, n), -1, dtype=np.int32)
        rows = np.zeros(log_cap, dtype=np.int32)
        ims = np.zeros(max(log_cap, 1), dtype=np.float32)
        st = J.GenStats(0, _i32p(acc), _i32p(rows), log_cap, 0.0, 0.0, 0, _f32p(ims) if log_cap > 0 else None)
        if traj is not None:
            st.traj = traj.data_ptr()
            st.traj_rows = traj_rows
            st.traj_cap = traj.numel() // (2 + 5 * traj_rows)
        self._c(self.lib.jf_generate(self.h, n, arr, _i32p(lens), C.byref(gp), _i32p(out), C.byref(st)))
        it = st.iterations
        k = min(it, log_cap)
        return GenOut(out, acc[:k], rows[:k], it, st.prefill_ms, st.decode_ms, st.kernel_launches, ims[:k],
                      st.traj_iters)

    def generate_device(self, d_prompts, prompt_lens, gen: Gen, d_out, d_truth=None, truth_len=0,
                        log_cap: int = 0):
        """Device buffers (torch int32 CUDA tensors) in and out (jf_generate_device)."""
        lens = np.ascontiguousarray(prompt_lens, dtype=np.int32)
        gp = gen.c_struct(d_truth.data_ptr() if d_truth is not None else None, truth_len)
        n = lens.size
        acc = np.full((max(log_cap, 1), n), -1, dtype=np.int32)
        rows = np.zeros(max(log_cap, 1), dtype=np.int32)
        ims = np.zeros(max(log_cap, 1), dtype=np.float32)
        st = J.GenStats(0, _i32p(acc), _i32p(rows), log_cap, 0.0, 0.0, 0, _f32p(ims) if log_cap > 0 else None)
        self._c(self.lib.jf_generate_device(self.h, n, d_prompts.data_ptr(), _i32p(lens), C.byref(gp),
                                            d_out.data_ptr(), C.byref(st)))
        it = st.iterations
        k = min(it, log_cap)
        return GenOut(None, acc[:k], rows[:k], it, st.prefill_ms, st.decode_ms, st.kernel_launches, ims[:k])

    def set_profiling(self, on: bool):
        self._c(self.lib.jf_set_profiling(self.h, 1 if on else 0))

    def kernel_time(self, cls: int):
        ms = C.c_double()
        n = C.c_longlong()
        self._c(self.lib.jf_kernel_time(self.h, cls, C.byref(ms), C.byref(n)))
        return ms.value, n.value

    def set_wait_limit(self, limit_ns: int):
        """Limit of every bounded device wait of this context (jf_set_wait_limit)."""
        self._c(self.lib.jf_set_wait_limit(self.h, int(limit_ns)))

    def wait_limit_probe(self):
        """(status, waited ns) of jf_wait_limit_probe; JF_ETIMEOUT is its expected status."""
        w = C.c_uint64()
        st = self.lib.jf_wait_limit_probe(self.h, C.byref(w))
        return st, w.value


def op_gemm(W, X, k_splits: int = 0, stream=None):
    """Y = X W^T through jf_op_gemm (torch CUDA tensors W [N,K], X [M,K], bf16 or fp32)."""
    import torch

    lib = J.load()
    N, K = W.shape
    M = X.shape[0]
    dtype = J.JF_BF16 if W.dtype == torch.bfloat16 else J.JF_F32
    nb = C.c_size_t()
    _check(lib, None, lib.jf_op_gemm_workspace_bytes(N, K, M, k_splits, C.byref(nb)))
    ws = torch.zeros(max(nb.value, 16), dtype=torch.uint8, device=W.device)
    err = torch.zeros(1, dtype=torch.int32, device=W.device)
    Y = torch.empty((M, N), dtype=torch.float32, device=W.device)
    s = stream if stream is not None else torch.cuda.current_stream()
    _check(lib, None, lib.jf_op_gemm(dtype, W.data_ptr(), X.data_ptr(), Y.data_ptr(), N, K, M, k_splits,
                                     ws.data_ptr(), nb.value, err.data_ptr(), s.cuda_stream))
    return Y, err, ws


def op_gemm_noalloc(W, X, k_splits: int = 0, stream=None):
    """Y = X W^T through jf_op_gemm_noalloc: bf16 only, no workspace argument (the library's fixed
    device scratch serves the split-K partials). Returns (Y, err_word, status)."""
    import torch

    lib = J.load()
    N, K = W.shape
    M = X.shape[0]
    err = torch.zeros(1, dtype=torch.int32, device=W.device)
    Y = torch.empty((M, N), dtype=torch.float32, device=W.device)
    s = stream if stream is not None else torch.cuda.current_stream()
    status = lib.jf_op_gemm_noalloc(W.data_ptr(), X.data_ptr(), Y.data_ptr(), N, K, M, k_splits, err.data_ptr(),
                                    s.cuda_stream)
    return Y, err, status


def trajectory_noisy_blocks(traj, n_iters: int, traj_rows: int, seq: int, new_tokens, prompt_len: int,
                            block_size: int, window: int, stream=None):
    """App. C training points of one sequence (jf_trajectory_noisy_blocks): traj and new_tokens are
    device int32 tensors; returns (noisy tokens [blocks, block_size], point index [blocks]) as device
    tensors."""
    import torch

    lib = J.load()
    n_new = new_tokens.numel()
    blocks = n_new // block_size
    noisy = torch.full((max(blocks, 1), block_size), -1, dtype=torch.int32, device=traj.device)
    point = torch.full((max(blocks, 1),), -1, dtype=torch.int32, device=traj.device)
    s = stream if stream is not None else torch.cuda.current_stream()
    _check(lib, None, lib.jf_trajectory_noisy_blocks(traj.data_ptr(), n_iters, traj_rows, seq, new_tokens.data_ptr(),
                                                     n_new, prompt_len, block_size, window, noisy.data_ptr(),
                                                     point.data_ptr(), s.cuda_stream))
    return noisy[:blocks], point[:blocks]
