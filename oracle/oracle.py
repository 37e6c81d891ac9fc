"""ctypes wrapper of the CPU oracle (TEST INFRASTRUCTURE ONLY).

Only the tests, `__graft_entry__.smoke()` and the CPU-baseline leg of `bench.py` may import
this module. The CUDA path never does, and this module never imports the CUDA path.

The model is the causal decoder of Jacobi Forcing (arXiv 2512.14681) Sec. 2.1, Eq. 1-3, in
the Qwen2.5 shape of Sec. 4.1; see jf_oracle.c for the arithmetic.
"""
from __future__ import annotations

import ctypes as C
from dataclasses import dataclass

import numpy as np

from . import build as _build

_lib = None


def lib():
    """Load (building first if needed) oracle/_build/libjforacle.so."""
    global _lib
    if _lib is None:
        path = _build.build()
        L = C.CDLL(path)
        vp, i32, i64, u64, dbl = C.c_void_p, C.c_int, C.c_long, C.c_uint64, C.c_double
        P = C.POINTER
        L.orc_sm64.restype = u64
        L.orc_sm64.argtypes = [u64, u64]
        L.orc_normal.restype = dbl
        L.orc_normal.argtypes = [u64, u64, u64]
        L.orc_round_bf16.restype = dbl
        L.orc_round_bf16.argtypes = [dbl]
        L.orc_model_create.restype = vp
        L.orc_model_create.argtypes = [vp]
        L.orc_model_free.argtypes = [vp]
        L.orc_init_random.argtypes = [vp, u64, dbl]
        L.orc_set_tensor.restype = i32
        L.orc_set_tensor.argtypes = [vp, i32, P(dbl), i64]
        L.orc_get_tensor.restype = i32
        L.orc_get_tensor.argtypes = [vp, i32, i64, i64, P(dbl)]
        L.orc_tensor_shape.restype = i32
        L.orc_tensor_shape.argtypes = [vp, i32, P(i64), P(i64)]
        L.orc_rmsnorm.argtypes = [i32, P(dbl), P(dbl), dbl, P(dbl)]
        L.orc_rope.argtypes = [i32, dbl, i64, P(dbl)]
        L.orc_silu.restype = dbl
        L.orc_silu.argtypes = [dbl]
        L.orc_linear_f64.argtypes = [i32, i32, i32, P(dbl), P(dbl), P(dbl)]
        L.orc_attend.argtypes = [i32, i32, i32, i32, P(dbl), P(P(dbl)), P(P(dbl)), P(C.c_ubyte), P(dbl)]
        L.orc_argmax_f32.restype = i32
        L.orc_argmax_f32.argtypes = [i32, P(dbl), P(C.c_float)]
        L.orc_cache_create.restype = vp
        L.orc_cache_create.argtypes = [vp, i32, i32]
        L.orc_cache_free.argtypes = [vp]
        L.orc_cache_len.restype = i32
        L.orc_cache_len.argtypes = [vp]
        L.orc_cache_truncate.restype = i32
        L.orc_cache_truncate.argtypes = [vp, i32]
        L.orc_commit.restype = i32
        L.orc_commit.argtypes = [vp, i32, P(C.c_int32)]
        L.orc_cache_entry.restype = i32
        L.orc_cache_entry.argtypes = [vp, i32, i32, i32, P(dbl)]
        L.orc_forward.restype = i32
        L.orc_forward.argtypes = [vp, vp, i32, P(C.c_int32), P(C.c_int32), P(C.c_int32), P(C.c_uint32), i32,
                                  P(C.c_int32), P(C.c_float), P(dbl), P(dbl)]
        L.orc_set_perturbation.argtypes = [dbl, u64]
        L.orc_num_threads.restype = i32
        L.orc_set_num_threads.argtypes = [i32]
        _lib = L
    return _lib


def _p(a, ct):
    return a.ctypes.data_as(C.POINTER(ct)) if a is not None else None


# ------------------------------------------------------------------------------------------
# Model configuration (Sec. 4.1 names the Qwen2.5 family; shapes come from the workloads)
# ------------------------------------------------------------------------------------------
class _Cfg(C.Structure):
    _fields_ = [("n_layers", C.c_int), ("d_model", C.c_int), ("n_heads", C.c_int), ("n_kv_heads", C.c_int),
                ("head_dim", C.c_int), ("d_ff", C.c_int), ("vocab", C.c_int), ("rms_eps", C.c_double),
                ("rope_theta", C.c_double), ("bf16", C.c_int), ("qkv_bias", C.c_int), ("tie_embeddings", C.c_int)]


@dataclass(frozen=True)
class ModelConfig:
    n_layers: int
    d_model: int
    n_heads: int
    n_kv_heads: int
    head_dim: int
    d_ff: int
    vocab: int
    rms_eps: float = 1e-6
    rope_theta: float = 1e4
    bf16: bool = False
    qkv_bias: bool = False        # per-feature biases on the Q, K, V projections (Qwen2.5 architecture)
    tie_embeddings: bool = False  # LM head = embedding matrix

    def c_struct(self) -> _Cfg:
        return _Cfg(self.n_layers, self.d_model, self.n_heads, self.n_kv_heads, self.head_dim, self.d_ff,
                    self.vocab, self.rms_eps, self.rope_theta, int(self.bf16), int(self.qkv_bias),
                    int(self.tie_embeddings))


# Logical tensor ids (jf_oracle.c): 0 embedding, 1 LM head (absent when tied), 2 final-norm gain;
# layer l at 8+16l: +0 attn-norm gain, +1 Wq, +2 Wk, +3 Wv, +4 Wo, +5 mlp-norm gain, +6 W_gate,
# +7 W_up, +8 W_down, and with QKV biases +9 b_q, +10 b_k, +11 b_v.
T_EMBED, T_LMHEAD, T_FNORM = 0, 1, 2
L_ANORM, L_WQ, L_WK, L_WV, L_WO, L_MNORM, L_WG, L_WU, L_WD, L_BQ, L_BK, L_BV = range(12)


def layer_tid(layer: int, w: int) -> int:
    return 8 + 16 * layer + w


class Model:
    """Oracle model: weights held at the model's storage precision (fp32, or bf16 values)."""

    def __init__(self, cfg: ModelConfig):
        self.cfg = cfg
        self._cs = cfg.c_struct()
        self.h = lib().orc_model_create(C.byref(self._cs))
        if not self.h:
            raise MemoryError("orc_model_create failed")

    def __del__(self):
        if getattr(self, "h", None):
            lib().orc_model_free(self.h)
            self.h = None

    def init_random(self, seed: int, std: float = 0.02) -> "Model":
        lib().orc_init_random(self.h, seed, std)
        return self

    def shape(self, tid: int):
        r, k = C.c_long(), C.c_long()
        if lib().orc_tensor_shape(C.byref(self._cs), tid, C.byref(r), C.byref(k)) != 0:
            raise ValueError(f"bad tensor id {tid}")
        return r.value, k.value

    def set_tensor(self, tid: int, values) -> None:
        a = np.ascontiguousarray(values, dtype=np.float64).ravel()
        if lib().orc_set_tensor(self.h, tid, _p(a, C.c_double), a.size) != 0:
            raise ValueError("orc_set_tensor failed")

    def get_tensor(self, tid: int, start: int = 0, count: int | None = None) -> np.ndarray:
        r, k = self.shape(tid)
        if count is None:
            count = r * k - start
        out = np.empty(count, dtype=np.float64)
        if lib().orc_get_tensor(self.h, tid, start, count, _p(out, C.c_double)) != 0:
            raise ValueError("orc_get_tensor failed")
        return out


class Cache:
    """Exact KV cache of the committed prefix of one sequence, plus the in-flight K/V."""

    def __init__(self, model: Model, max_ctx: int, max_rows: int):
        self.model = model
        self.h = lib().orc_cache_create(model.h, max_ctx, max_rows)
        if not self.h:
            raise MemoryError("orc_cache_create failed")

    def __del__(self):
        if getattr(self, "h", None):
            lib().orc_cache_free(self.h)
            self.h = None

    def __len__(self):
        return lib().orc_cache_len(self.h)

    def truncate(self, n: int) -> None:
        if lib().orc_cache_truncate(self.h, n) != 0:
            raise ValueError("truncate beyond length")

    def commit(self, rows) -> None:
        r = np.ascontiguousarray(rows, dtype=np.int32)
        if lib().orc_commit(self.h, r.size, _p(r, C.c_int32)) != 0:
            raise ValueError("orc_commit failed")

    def entry(self, layer: int, which: int, pos: int) -> np.ndarray:
        c = self.model.cfg
        out = np.empty(c.n_kv_heads * c.head_dim, dtype=np.float64)
        if lib().orc_cache_entry(self.h, layer, which, pos, _p(out, C.c_double)) != 0:
            raise ValueError("orc_cache_entry failed")
        return out.reshape(c.n_kv_heads, c.head_dim)


@dataclass
class ForwardOut:
    argmax: np.ndarray          # int32 [M]
    top2: np.ndarray            # float32 [M, 2] (largest, second largest logit, fp32)
    logits: np.ndarray | None   # float64 [M, V]
    hidden: np.ndarray | None   # float64 [M, d] final residual stream

    @property
    def margin(self) -> np.ndarray:
        return (self.top2[:, 0].astype(np.float64) - self.top2[:, 1].astype(np.float64))


def forward(model: Model, cache: Cache, tokens, pos, seg=None, anc=None, want_logits=False,
            want_hidden=False) -> ForwardOut:
    """One forward over in-flight rows (Eq. 3; mask rule of Sec. 3.2 / Algorithm 1)."""
    t = np.ascontiguousarray(tokens, dtype=np.int32)
    M = t.size
    p = np.ascontiguousarray(pos, dtype=np.int32)
    s = np.zeros(M, dtype=np.int32) if seg is None else np.ascontiguousarray(seg, dtype=np.int32)
    n_seg = int(s.max()) + 1 if M else 1
    a = np.zeros(n_seg, dtype=np.uint32) if anc is None else np.ascontiguousarray(anc, dtype=np.uint32)
    am = np.empty(M, dtype=np.int32)
    top2 = np.empty((M, 2), dtype=np.float32)
    logits = np.empty((M, model.cfg.vocab), dtype=np.float64) if want_logits else None
    hidden = np.empty((M, model.cfg.d_model), dtype=np.float64) if want_hidden else None
    rc = lib().orc_forward(model.h, cache.h, M, _p(t, C.c_int32), _p(p, C.c_int32), _p(s, C.c_int32),
                           _p(a, C.c_uint32), a.size, _p(am, C.c_int32), _p(top2, C.c_float),
                           _p(logits, C.c_double), _p(hidden, C.c_double))
    if rc != 0:
        raise ValueError(f"orc_forward failed ({rc})")
    return ForwardOut(am, top2, logits, hidden)


# ------------------------------------------------------------------------------------------
# Building blocks, exported for the pins
# ------------------------------------------------------------------------------------------
def sm64(state: int, i: int) -> int:
    return int(lib().orc_sm64(state & (2**64 - 1), i & (2**64 - 1)))


def normal(seed: int, tid: int, e: int) -> float:
    return float(lib().orc_normal(seed, tid, e))


def round_bf16(x: float) -> float:
    return float(lib().orc_round_bf16(float(x)))


def rmsnorm(x, gain, eps):
    x = np.ascontiguousarray(x, dtype=np.float64)
    g = np.ascontiguousarray(gain, dtype=np.float64)
    y = np.empty_like(x)
    lib().orc_rmsnorm(x.size, _p(x, C.c_double), _p(g, C.c_double), eps, _p(y, C.c_double))
    return y


def rope(v, pos, theta):
    v = np.array(v, dtype=np.float64)
    lib().orc_rope(v.size, theta, pos, _p(v, C.c_double))
    return v


def silu(x: float) -> float:
    return float(lib().orc_silu(float(x)))


def linear(x, W):
    x = np.ascontiguousarray(x, dtype=np.float64)
    W = np.ascontiguousarray(W, dtype=np.float64)
    M, K = x.shape
    N = W.shape[0]
    y = np.empty((M, N), dtype=np.float64)
    lib().orc_linear_f64(M, N, K, _p(x, C.c_double), _p(W, C.c_double), _p(y, C.c_double))
    return y


def attend(q, keys, values, visible, n_kv_heads):
    """q [Hq, hd]; keys/values [n, Hkv, hd]; visible [n] -> out [Hq, hd]."""
    q = np.ascontiguousarray(q, dtype=np.float64)
    Hq, hd = q.shape
    keys = np.ascontiguousarray(keys, dtype=np.float64)
    values = np.ascontiguousarray(values, dtype=np.float64)
    n = keys.shape[0]
    kp = (C.POINTER(C.c_double) * max(n, 1))()
    vp = (C.POINTER(C.c_double) * max(n, 1))()
    for j in range(n):
        kp[j] = C.cast(keys[j].ctypes.data, C.POINTER(C.c_double))
        vp[j] = C.cast(values[j].ctypes.data, C.POINTER(C.c_double))
    vis = np.ascontiguousarray(visible, dtype=np.uint8)
    out = np.empty((Hq, hd), dtype=np.float64)
    lib().orc_attend(Hq, n_kv_heads, hd, n, _p(q, C.c_double), kp, vp, _p(vis, C.c_ubyte), _p(out, C.c_double))
    return out


def argmax_f32(logits):
    x = np.ascontiguousarray(logits, dtype=np.float64)
    t2 = np.empty(2, dtype=np.float32)
    a = lib().orc_argmax_f32(x.size, _p(x, C.c_double), _p(t2, C.c_float))
    return int(a), t2


def num_threads() -> int:
    return int(lib().orc_num_threads())


def set_num_threads(n: int) -> None:
    lib().orc_set_num_threads(n)


def set_perturbation(eps: float, seed: int = 0) -> None:
    """Rounding-noise diagnostic of jf_oracle.c (off when eps = 0): every value is scaled by
    (1 + eps * u), u uniform in [-1, 1), just before its bf16 rounding point."""
    lib().orc_set_perturbation(float(eps), seed & (2**64 - 1))
