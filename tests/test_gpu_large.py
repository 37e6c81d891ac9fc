"""Full-size parity (Qwen2.5-1.5B and -7B shapes, bf16) in the launch configuration the bench uses.

At these sizes the oracle is used on samples it can compute one by one (weights, a short greedy
continuation), and the rest is checked through properties that hold at any size:
* greedy Jacobi decoding reproduces greedy AR decoding token for token (Sec. 2.1, Eq. 3);
* with draft injection against the true greedy continuation, iteration i commits exactly
  1 + (number of leading uncorrupted draft tokens), the corruption decisions coming from the
  oracle's own implementation of the injection rule.
"""
import os

import numpy as np
import pytest

from oracle import jacobi as OJ
from oracle import oracle as O
from paper_2512_14681_gb300 import inputs as I
from tests.parity import compare_with_resync, need_gpu, wide_logit_tol

pytestmark = pytest.mark.gpu


def _round(shape, v):
    return O.round_bf16(v) if shape.bf16 else float(np.float32(v))


def _sampled_weights(ctx, shape, n=64):
    rng = np.random.default_rng(5)
    head = [0] if shape.tie_embeddings else [0, 1]  # a tied model has no separate LM head
    per = (1, 2, 3, 4, 6, 7, 8) + ((9, 10, 11) if shape.qkv_bias else ())
    tids = head + [8 + 16 * l + w for l in (0, shape.n_layers - 1) for w in per]
    bad = 0
    for tid in tids:
        rows, cols = _shape_of(shape, tid)
        for e in rng.integers(0, rows * cols, size=n):
            ref = _round(shape, I.WEIGHT_STD * O.normal(I.WEIGHT_SEED, tid, int(e)))
            got = float(ctx.get_weights(tid, int(e), 1)[0])
            bad += got != ref
    assert bad <= 1


def _shape_of(shape, tid):
    d, qd, kvd = shape.d_model, shape.n_heads * shape.head_dim, shape.n_kv_heads * shape.head_dim
    if tid in (0, 1):
        return shape.vocab, d
    w = (tid - 8) % 16
    return {1: (qd, d), 2: (kvd, d), 3: (kvd, d), 4: (d, qd), 6: (shape.d_ff, d), 7: (shape.d_ff, d),
            8: (d, shape.d_ff), 9: (1, qd), 10: (1, kvd), 11: (1, kvd)}[w]


def _expected_inject_counts(truth, P0, n, p, seed, vocab, max_new):
    """Block-mode injected acceptance: k = 1 + leading uncorrupted draft positions."""
    T = OJ.inject_threshold(p)
    counts, P, it, start = [], P0, 0, P0
    while P - P0 < max_new:
        L = start + n - P
        k = 1
        while k < L and OJ.inject_token(seed, P + k, it, truth[P + k - P0], T, vocab) == truth[P + k - P0]:
            k += 1
        counts.append(k)
        P += k
        it += 1
        if P >= start + n:
            start = P
    return counts


_ORACLE_MODELS = {}


def _host_memory_ok(shape) -> bool:
    need = shape.weight_bytes() + (8 << 30)
    try:
        avail = os.sysconf("SC_AVPHYS_PAGES") * os.sysconf("SC_PAGE_SIZE")
    except (ValueError, OSError):
        avail = 0
    return avail >= need or shape.name in _ORACLE_MODELS


def _oracle_model(shape):
    """The full-size oracle model, drawn once per shape and shared by this module's tests."""
    if shape.name not in _ORACLE_MODELS:
        _ORACLE_MODELS.clear()  # at most one full-size model in host memory at a time
        _ORACLE_MODELS[shape.name] = O.Model(O.ModelConfig(**shape.oracle_kwargs())).init_random(
            I.WEIGHT_SEED, I.WEIGHT_STD)
    return _ORACLE_MODELS[shape.name]


@pytest.fixture(scope="module", params=[I.QWEN15B_BF16, I.QWEN7B_BF16], ids=lambda s: s.name)
def big(request):
    torch = need_gpu()
    from paper_2512_14681_gb300.jacobi import Context

    shape = request.param
    free, total = torch.cuda.mem_get_info()
    if free < shape.weight_bytes() * 1.3:
        pytest.skip("not enough device memory")
    ctx = Context(shape, max_seqs=1, max_ctx=2048, max_rows=64, logits_rows=32)
    ctx.init_random_weights(I.WEIGHT_SEED, I.WEIGHT_STD)
    yield shape, ctx
    ctx.close()


def test_sampled_weights_equal_oracle(big):
    shape, ctx = big
    _sampled_weights(ctx, shape)


def test_jacobi_equals_ar_full_size(big):
    shape, ctx = big
    from paper_2512_14681_gb300.jacobi import Gen

    n = 16 if shape is I.QWEN15B_BF16 else 32
    prompt = I.prompt_tokens(shape.vocab, 512 if n == 16 else 1024)
    ar = ctx.generate([prompt], Gen(mode="ar", max_new=64)).tokens[0]
    jac = ctx.generate([prompt], Gen(block_size=n, max_new=64)).tokens[0]
    assert np.array_equal(ar, jac)


def test_injected_counts_full_size(big):
    shape, ctx = big
    from paper_2512_14681_gb300.jacobi import Gen

    n, p = (16, 0.5) if shape is I.QWEN15B_BF16 else (32, 0.3)
    prompt = I.prompt_tokens(shape.vocab, 512 if n == 16 else 1024)
    max_new = 96
    truth = ctx.generate([prompt], Gen(mode="ar", max_new=max_new + n + n + 1)).tokens[0]
    out = ctx.generate([prompt], Gen(block_size=n, init="inject", inject_p=p, seed=I.INJECT_SEED, max_new=max_new),
                       truth=np.array([truth], dtype=np.int32))
    assert np.array_equal(out.tokens[0], truth[:max_new])
    exp = _expected_inject_counts(truth.tolist(), prompt.size, n, p, I.INJECT_SEED, shape.vocab, max_new)
    assert out.counts[:, 0].tolist() == exp


def test_short_greedy_continuation_matches_oracle(big):
    """The oracle decodes a short continuation of a short prompt on the full-size model."""
    shape, ctx = big
    from paper_2512_14681_gb300.jacobi import Gen

    if not _host_memory_ok(shape):
        pytest.skip("not enough host memory for the full-size oracle")
    prompt = I.prompt_tokens(shape.vocab, 16, seed=31)
    new = 6 if shape is I.QWEN7B_BF16 else 12
    model = _oracle_model(shape)

    def run_oracle(p, max_new, offset):
        return OJ.generate_jacobi(model, p, OJ.GenParams(block_size=4, max_new=max_new))

    def run_gpu(p, max_new, offset):
        out = ctx.generate([p], Gen(block_size=4, max_new=max_new))
        return out.tokens[0], out.counts[:, 0]

    compare_with_resync(run_gpu, run_oracle, prompt, new, True, max_flags=1)


def test_full_depth_logits_match_oracle(big):
    """Every layer of the full-size model: the fp32 logits of a 32-row causal forward over a short
    committed cache (Eq. 3), element by element against the oracle (bf16 model: the larger of 3e-2
    and twice the spread one fp32 unit at every bf16 rounding point gives the oracle's own logits
    through all 28 layers), and the greedy decisions outside flagged near-ties."""
    shape, ctx = big
    if not _host_memory_ok(shape):
        pytest.skip("not enough host memory for the full-size oracle")
    model = _oracle_model(shape)
    prompt = I.prompt_tokens(shape.vocab, 20, seed=33)
    rows = I.prompt_tokens(shape.vocab, 32, seed=34)
    if ctx.seq_len(0):
        ctx.truncate(0, 0)
    ctx.prefill(0, prompt)
    lg, hid, am = ctx.forward_logits(0, rows)
    ctx.truncate(0, 0)
    oc = O.Cache(model, 64, 32)
    O.forward(model, oc, prompt, np.arange(20))
    oc.commit(np.arange(20))
    ref = O.forward(model, oc, rows, np.arange(20, 52), want_logits=True, want_hidden=True)
    case = "full-7b-32rows" if shape is I.QWEN7B_BF16 else "full-1.5b-32rows"
    tol, sd_tol = wide_logit_tol(case)
    diff = np.abs(lg - ref.logits)
    assert diff.max() <= tol, f"logit max-abs diff {diff.max()} (bound {tol})"
    assert diff.std() <= sd_tol, f"logit diff std {diff.std()} (bound {sd_tol})"
    assert np.all((am == ref.argmax) | (ref.margin < 2 * tol))
