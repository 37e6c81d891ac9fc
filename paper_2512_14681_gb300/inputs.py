"""Seeded synthetic inputs shared by the CUDA path's tests, the oracle's tests and the bench.

Holds none of the method's arithmetic: model shapes, seeds and prompt tokens only. The paper's
workloads (HumanEval, MBPP, GSM8K, MATH on trained Qwen2.5 checkpoints) are not available, so
uniform-random prompts over the vocabulary and N(0, 0.02) random weights of the same shapes
stand in for them. Weights are not generated here: each side draws them from the same
counter-based generator definition (SplitMix64 + Box-Muller, keyed by seed, tensor id and
element index).
"""
from __future__ import annotations

from dataclasses import dataclass

import numpy as np


@dataclass(frozen=True)
class ModelShape:
    name: str
    n_layers: int
    d_model: int
    n_heads: int
    n_kv_heads: int
    head_dim: int
    d_ff: int
    vocab: int
    rms_eps: float
    rope_theta: float
    bf16: bool
    qkv_bias: bool = False        # per-feature biases on the Q, K, V projections
    tie_embeddings: bool = False  # the LM head is the embedding matrix

    def oracle_kwargs(self) -> dict:
        return dict(n_layers=self.n_layers, d_model=self.d_model, n_heads=self.n_heads,
                    n_kv_heads=self.n_kv_heads, head_dim=self.head_dim, d_ff=self.d_ff, vocab=self.vocab,
                    rms_eps=self.rms_eps, rope_theta=self.rope_theta, bf16=self.bf16, qkv_bias=self.qkv_bias,
                    tie_embeddings=self.tie_embeddings)

    def weight_bytes(self) -> int:
        """Bytes of every weight matrix read by one forward pass (embedding rows excluded)."""
        es = 2 if self.bf16 else 4
        d, hd = self.d_model, self.head_dim
        per_layer = d * (self.n_heads + 2 * self.n_kv_heads) * hd + self.n_heads * hd * d + 3 * d * self.d_ff
        if self.qkv_bias:
            per_layer += (self.n_heads + 2 * self.n_kv_heads) * hd
        return es * (self.n_layers * per_layer + self.vocab * d) + 4 * d * (2 * self.n_layers + 1)

    def kv_bytes_per_token(self) -> int:
        es = 2 if self.bf16 else 4
        return 2 * self.n_layers * self.n_kv_heads * self.head_dim * es


# Tiny fp32 decoder: 2 layers, d 256, 4/2 heads of 64, SwiGLU 1024, vocab 4096, theta 1e4.
TINY_F32 = ModelShape("tiny-f32", 2, 256, 4, 2, 64, 1024, 4096, 1e-6, 1e4, False)
# Small bf16 decoder spanning several GEMM tiles (parity at sizes the oracle finishes quickly).
SMALL_BF16 = ModelShape("small-bf16", 2, 512, 8, 2, 128, 1536, 8192, 1e-6, 1e6, True)
# The tiny and small decoders with per-feature Q/K/V biases and tied embeddings (the Qwen2.5
# architecture's options), for parity of those paths.
TINY_F32_BT = ModelShape("tiny-f32-bias-tied", 2, 256, 4, 2, 64, 1024, 4096, 1e-6, 1e4, False, True, True)
SMALL_BF16_BT = ModelShape("small-bf16-bias-tied", 2, 512, 8, 2, 128, 1536, 8192, 1e-6, 1e6, True, True, True)
# Qwen2.5-1.5B shape, bf16 (Q/K/V biases and tied embeddings, as in that architecture).
QWEN15B_BF16 = ModelShape("qwen2.5-1.5b-shape-bf16", 28, 1536, 12, 2, 128, 8960, 151936, 1e-6, 1e6, True, True, True)
# Qwen2.5-7B shape, bf16 (Q/K/V biases, untied LM head, as in that architecture).
QWEN7B_BF16 = ModelShape("qwen2.5-7b-shape-bf16", 28, 3584, 28, 4, 128, 18944, 152064, 1e-6, 1e6, True, True)

# Two layers of the Qwen2.5-7B shape (every per-layer width and the full vocabulary of the 7B model), so
# that the oracle can check forwards at the 7B widths in seconds.
QWEN7B_2L_BF16 = ModelShape("qwen2.5-7b-shape-2layer-bf16", 2, 3584, 28, 4, 128, 18944, 152064, 1e-6, 1e6, True,
                            True)

SHAPES = {s.name: s for s in (TINY_F32, SMALL_BF16, TINY_F32_BT, SMALL_BF16_BT, QWEN15B_BF16, QWEN7B_BF16,
                              QWEN7B_2L_BF16)}

WEIGHT_SEED = 0
WEIGHT_STD = 0.02
PROMPT_SEED = 1
INJECT_SEED = 2


def prompt_tokens(vocab: int, length: int, seed: int = PROMPT_SEED) -> np.ndarray:
    """Uniform-random prompt tokens over [0, vocab) (numpy PCG64 seeded with `seed`)."""
    rng = np.random.default_rng(seed)
    return rng.integers(0, vocab, size=length, dtype=np.int64).astype(np.int32)


def random_array(shape, seed: int, scale: float = 1.0, dtype=np.float32) -> np.ndarray:
    """Standard-normal test array (numpy PCG64), used for kernel-level parity inputs."""
    rng = np.random.default_rng(seed)
    return (rng.standard_normal(shape) * scale).astype(dtype)
