"""Attention over long committed contexts (Sec. 2.1, Eq. 3 over the exact KV cache).

With more than 8 x 128 committed keys every chunk lane of the bf16 attention walks several
chunks (online softmax across chunks, next chunk prefetched), and the lane fold runs on
partial states. Checked here:
* small bf16 model, 2540 committed tokens + 37 in-flight rows crossing a 128-key chunk
  boundary: logits against the oracle (3e-2), argmax equal outside flagged near-ties;
* a batch of three sequences with different long prompts decodes exactly as each one alone
  (a row's arithmetic does not depend on the rows in flight with it);
* greedy Jacobi decoding equals greedy AR decoding on the device at 2540 committed tokens
  (small model) and at 16384 committed tokens (1.5B shape), and with a 256-row window whose
  attention runs the unclustered form of the kernel.
"""
import numpy as np
import pytest

from oracle import oracle as O
from paper_2512_14681_gb300 import inputs as I
from tests.parity import LOGIT_TOL, need_gpu

pytestmark = pytest.mark.gpu

P_LONG = 2540  # 20 chunks of 128 keys: lanes 0-3 hold three chunks, lanes 4-7 two


@pytest.fixture(scope="module")
def small():
    need_gpu()
    from paper_2512_14681_gb300.jacobi import Context

    shape = I.SMALL_BF16
    ctx = Context(shape, max_seqs=3, max_ctx=3072, max_rows=128, logits_rows=48)
    ctx.init_random_weights(I.WEIGHT_SEED, I.WEIGHT_STD)
    yield shape, ctx
    ctx.close()


def test_long_cache_logits_match_oracle(small):
    shape, ctx = small
    model = O.Model(O.ModelConfig(**shape.oracle_kwargs())).init_random(I.WEIGHT_SEED, I.WEIGHT_STD)
    toks = I.prompt_tokens(shape.vocab, P_LONG + 37, seed=51)
    ctx.truncate(0, 0) if ctx.seq_len(0) else None
    q0 = ctx.prefill(0, toks[:P_LONG])
    oc = O.Cache(model, 3072, P_LONG)
    pre = O.forward(model, oc, toks[:P_LONG], np.arange(P_LONG))
    oc.commit(np.arange(P_LONG))
    tol = LOGIT_TOL[shape.bf16]
    assert q0 == pre.argmax[-1] or pre.margin[-1] < 2 * tol
    lg, _, am = ctx.forward_logits(0, toks[P_LONG:])
    ref = O.forward(model, oc, toks[P_LONG:], np.arange(P_LONG, P_LONG + 37), want_logits=True)
    d = np.abs(lg - ref.logits).max()
    assert d <= tol, f"logit max-abs diff over a {P_LONG}-token cache: {d}"
    flagged = ref.margin < 2 * tol
    assert np.all((am == ref.argmax) | flagged)
    ctx.truncate(0, 0)


def test_long_context_batch_equals_single(small):
    shape, ctx = small
    from paper_2512_14681_gb300.jacobi import Gen

    prompts = [I.prompt_tokens(shape.vocab, L, seed=60 + i) for i, L in enumerate((P_LONG, 1100, 2047))]
    gen = Gen(block_size=16, max_new=24)
    both = ctx.generate(prompts, gen)
    for i, p in enumerate(prompts):
        one = ctx.generate([p], gen)
        assert np.array_equal(both.tokens[i], one.tokens[0]), f"sequence {i} differs in a batch"


def test_long_context_jacobi_equals_ar(small):
    shape, ctx = small
    from paper_2512_14681_gb300.jacobi import Gen

    prompt = I.prompt_tokens(shape.vocab, P_LONG, seed=52)
    ar = ctx.generate([prompt], Gen(mode="ar", max_new=40)).tokens[0]
    for kw in (dict(block_size=16), dict(block_size=32, mode="window"),
               dict(block_size=8, n_blocks=3, pool_size=8, cand_per_iter=1)):
        jac = ctx.generate([prompt], Gen(max_new=40, **kw)).tokens[0]
        assert np.array_equal(jac, ar), f"{kw}: Jacobi output differs from AR at {P_LONG} cached tokens"


def test_jacobi_equals_ar_16k_context_1p5b():
    torch = need_gpu()
    from paper_2512_14681_gb300.jacobi import Context, Gen

    shape = I.QWEN15B_BF16
    free, _ = torch.cuda.mem_get_info()
    if free < shape.weight_bytes() * 1.5:
        pytest.skip("not enough device memory")
    P = 16384
    ctx = Context(shape, max_seqs=1, max_ctx=P + 128, max_rows=64)
    try:
        ctx.init_random_weights(I.WEIGHT_SEED, I.WEIGHT_STD)
        prompt = I.prompt_tokens(shape.vocab, P, seed=53)
        ar = ctx.generate([prompt], Gen(mode="ar", max_new=24)).tokens[0]
        jac = ctx.generate([prompt], Gen(block_size=16, max_new=24)).tokens[0]
        assert np.array_equal(jac, ar)
    finally:
        ctx.close()


def test_unclustered_attention_decodes_like_clustered():
    """A 256-row Jacobi window on the small model has 16 attention units (2 KV heads x 8 query
    tiles), more than the 15 8-CTA clusters of the attention kernel that a GB300 holds at once: as
    clusters they take two waves, as independent CTAs (128) one, so its forwards run the unclustered
    form (the last lane of a unit folds all its rows). AR forwards (one row, two units) run the
    clustered form. Both fold in lane order with the same arithmetic: the tokens are identical."""
    need_gpu()
    from paper_2512_14681_gb300.jacobi import Context, Gen

    shape = I.SMALL_BF16
    ctx = Context(shape, max_seqs=1, max_ctx=3072, max_rows=256, logits_rows=16)
    try:
        ctx.init_random_weights(I.WEIGHT_SEED, I.WEIGHT_STD)
        prompt = I.prompt_tokens(shape.vocab, P_LONG, seed=54)
        ar = ctx.generate([prompt], Gen(mode="ar", max_new=48)).tokens[0]
        out = ctx.generate([prompt], Gen(block_size=256, mode="window", max_new=48))
        assert out.rows.max() == 256
        assert np.array_equal(out.tokens[0], ar)
    finally:
        ctx.close()
