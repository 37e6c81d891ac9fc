"""Byte counts behind the bench's roofline, pinned to the model shapes' closed forms.

One Jacobi iteration streams every weight matrix once (q, k, v, o, gate, up, down per layer, the
Q/K/V biases, the LM head (the embedding matrix when tied), the fp32 norm gains) and reads the
committed K/V of every layer; the iteration's roofline
is those bytes over the HBM bandwidth. The figures below are the Qwen2.5 shapes' own sizes (7B:
3584 wide, 28 query / 4 KV heads of 128, SwiGLU 18944, vocabulary 152064, 28 layers; 1.5B: 1536,
12 / 2, 8960, 151936, 28).
"""
import bench
from paper_2512_14681_gb300 import inputs as I


def test_7b_layer_parameters_and_iteration_bytes():
    s = I.QWEN7B_BF16
    attn = 3584 * (28 + 2 * 4) * 128 + 28 * 128 * 3584        # q, k, v, o
    mlp = 3 * 3584 * 18944                                    # gate, up, down
    assert attn + mlp == 233_046_016                          # 233.05 M parameters a layer
    bias = (28 + 2 * 4) * 128                                 # q, k, v biases
    lm = 152064 * 3584
    assert s.weight_bytes() == 2 * (28 * (attn + mlp + bias) + lm) + 4 * 3584 * 57
    assert abs(s.weight_bytes() / 1e9 - 14.141) < 0.001


def test_kv_bytes_per_token():
    assert I.QWEN7B_BF16.kv_bytes_per_token() == 2 * 28 * 4 * 128 * 2 == 57_344
    assert I.QWEN15B_BF16.kv_bytes_per_token() == 2 * 28 * 2 * 128 * 2 == 28_672


def test_15b_iteration_bytes():
    s = I.QWEN15B_BF16
    per_layer = 1536 * (12 + 4) * 128 + 12 * 128 * 1536 + 3 * 1536 * 8960 + (12 + 4) * 128
    assert s.weight_bytes() == 2 * (28 * per_layer + 151936 * 1536) + 4 * 1536 * 57  # tied: the head is read once
    assert abs(s.weight_bytes() / 1e9 - 3.087) < 0.001


def test_bench_workloads_fit_their_context():
    """Every bench workload's in-flight rows and context fit the capacities bench.py requests."""
    for name, w in bench.WORKLOADS.items():
        g = w.ngram or w.block
        rows = w.blocks * w.block + w.cands * g
        assert rows <= 512, name   # one context of 512 rows serves the prefill chunks and every iteration
        assert w.blocks >= 1 and w.block >= 1 and w.new >= 1 and 0.0 <= w.p <= 1.0, name
        assert w.shape in I.SHAPES, name
    assert bench.DEFAULT_WORKLOAD in bench.WORKLOADS
    assert set(bench.ALIASES.values()) <= set(bench.WORKLOADS)
