"""Serving many sequences at once (batch up to 16): per-sequence block sizes and late joins whose
prompts are prefilled in chunks inside the decode iterations, beside the running sequences' Jacobi
rows.

The paper verifies drafts "by appending them along the batch dimension" (Sec. 3.2) and decodes each
sequence block by block (Eq. 4); sequences served together are independent, so each must decode
exactly as it does alone: the same tokens and the same committed count in every one of its
iterations. Each is also compared with the oracle's decoding loop (flagged near-ties re-synchronised).
"""
import numpy as np
import pytest

from oracle import jacobi as OJ
from oracle import oracle as O
from paper_2512_14681_gb300 import inputs as I
from tests.parity import compare_with_resync, need_gpu

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", params=[I.TINY_F32, I.SMALL_BF16], ids=lambda s: s.name)
def setup(request):
    need_gpu()
    from paper_2512_14681_gb300.jacobi import Context

    shape = request.param
    ctx = Context(shape, max_seqs=16, max_ctx=512, max_rows=192)
    ctx.init_random_weights(I.WEIGHT_SEED, I.WEIGHT_STD)
    model = O.Model(O.ModelConfig(**shape.oracle_kwargs())).init_random(I.WEIGHT_SEED, I.WEIGHT_STD)
    yield shape, ctx, model
    ctx.close()


def _own_counts(counts, b):
    c = counts[:, b]
    return c[c >= 0].tolist()


def _against_alone_and_oracle(shape, ctx, model, prompts, both, gens, max_new):
    from paper_2512_14681_gb300.jacobi import Gen

    for b, p in enumerate(prompts):
        g = gens[b]
        one = ctx.generate([p], g)
        assert np.array_equal(both.tokens[b], one.tokens[0]), f"sequence {b}: tokens differ from its own run"
        assert _own_counts(both.counts, b) == one.counts[:, 0].tolist(), f"sequence {b}: counts differ"
        kw = dict(block_size=g.block_size, n_blocks=g.n_blocks, spawn_ratio=g.spawn_ratio, pool_size=g.pool_size,
                  cand_per_iter=g.cand_per_iter, mode=g.mode)

        def run_oracle(pp, n_new, offset, kw=kw):
            return OJ.generate_jacobi(model, pp, OJ.GenParams(max_new=n_new, **kw))

        def run_gpu(pp, n_new, offset, g=g):
            out = ctx.generate([pp], Gen(**{**g.__dict__, "max_new": n_new}))
            return out.tokens[0], out.counts[:, 0]

        # the first segment compared is the batched run's own sequence
        first = [True]

        def run_gpu_first(pp, n_new, offset):
            if first[0]:
                first[0] = False
                return both.tokens[b], np.array(_own_counts(both.counts, b))
            return run_gpu(pp, n_new, offset)

        compare_with_resync(run_gpu_first, run_oracle, p, max_new, shape.bf16, max_flags=2)


def test_sixteen_sequences(setup):
    shape, ctx, model = setup
    from paper_2512_14681_gb300.jacobi import Gen

    prompts = [I.prompt_tokens(shape.vocab, 5 + 7 * b, seed=200 + b) for b in range(16)]
    gen = Gen(block_size=8, max_new=24)
    both = ctx.generate(prompts, gen)
    assert both.rows.max() == 16 * 8
    _against_alone_and_oracle(shape, ctx, model, prompts, both, [gen] * 16, 24)


def test_per_sequence_block_sizes(setup):
    """Six sequences with block sizes 1, 3, 4, 8, 12 and 16, multi-block with recycling."""
    shape, ctx, model = setup
    from paper_2512_14681_gb300.jacobi import Gen

    sizes = [1, 3, 4, 8, 12, 16]
    prompts = [I.prompt_tokens(shape.vocab, 9 + 5 * b, seed=300 + b) for b in range(len(sizes))]
    base = dict(n_blocks=2, spawn_ratio=0.5, pool_size=8, cand_per_iter=1, max_new=32)
    both = ctx.generate(prompts, Gen(block_size=16, block_sizes=tuple(sizes), **base))
    gens = [Gen(block_size=n, **base) for n in sizes]
    _against_alone_and_oracle(shape, ctx, model, prompts, both, gens, 32)


def test_late_joins_with_chunked_prefill(setup):
    """Four sequences, two of them joining at forwards 3 and 7 with prompts of 61 and 45 tokens
    prefilled 16 rows per forward beside the others' Jacobi rows; the trajectory record shows the
    chunks inside forwards that also carry other sequences' rows."""
    torch = need_gpu()
    shape, ctx, model = setup
    from paper_2512_14681_gb300.jacobi import Gen, trajectory_records

    prompts = [I.prompt_tokens(shape.vocab, L, seed=400 + L) for L in (20, 33, 61, 45)]
    gen = Gen(block_size=8, max_new=40, join_iters=(0, 0, 3, 7), prefill_chunk=16)
    R = 128
    buf = torch.zeros(256 * (2 + 5 * R), dtype=torch.int32, device="cuda")
    both = ctx.generate(prompts, gen, traj=buf, traj_rows=R)
    recs = trajectory_records(buf, both.traj_iters, R)
    for b, j in ((2, 3), (3, 7)):
        chunks = [(i, r) for i, r in enumerate(recs) if np.any((r["seq"] == b) & (r["kind"] == 3))]
        assert chunks[0][0] == j
        assert [int(t) for _, r in chunks for t in r["token"][r["seq"] == b]] == prompts[b].tolist()
        assert all(np.any(r["seq"] != b) for _, r in chunks)  # beside other sequences' rows
    gens = [Gen(block_size=8, max_new=40)] * 4
    _against_alone_and_oracle(shape, ctx, model, prompts, both, gens, 40)


def test_serving_parameters_are_checked(setup):
    shape, ctx, model = setup
    from paper_2512_14681_gb300 import _lib as J
    from paper_2512_14681_gb300.jacobi import Gen

    prompts = [I.prompt_tokens(shape.vocab, 10, seed=500 + b) for b in range(2)]
    bad = [Gen(block_size=8, block_sizes=(8, 9)),                 # larger than block_size
           Gen(block_size=8, block_sizes=(0, 8)),
           Gen(block_size=8, join_iters=(0, -1)),
           Gen(block_size=8, join_iters=(0, 2), prefill_chunk=1000)]  # chunk beyond max_rows
    for g in bad:
        with pytest.raises(J.JfError) as ei:
            ctx.generate(prompts, g)
        assert ei.value.status == J.JF_EINVAL


def test_max_segments_bounds_the_chains():
    """jf_runtime_config.max_segments: a context sized for 3 attention chains decodes one sequence
    with two recycled candidates a forward (3 chains) exactly as a default-sized one does, and
    refuses two such sequences (6 chains) with JF_ECAPACITY before any launch."""
    need_gpu()
    from paper_2512_14681_gb300 import _lib as J
    from paper_2512_14681_gb300.jacobi import Context, Gen

    shape = I.SMALL_BF16
    gen = Gen(block_size=8, pool_size=16, cand_per_iter=2, max_new=32)
    prompts = [I.prompt_tokens(shape.vocab, 24, seed=90 + i) for i in range(2)]
    ref = Context(shape, max_seqs=2, max_ctx=256, max_rows=64)
    small = Context(shape, max_seqs=2, max_ctx=256, max_rows=64, max_segments=3)
    try:
        for c in (ref, small):
            c.init_random_weights(I.WEIGHT_SEED, I.WEIGHT_STD)
        a = ref.generate([prompts[0]], gen)
        b = small.generate([prompts[0]], gen)
        assert np.array_equal(a.tokens, b.tokens) and np.array_equal(a.counts, b.counts)
        with pytest.raises(J.JfError) as ei:
            small.generate(prompts, gen)
        assert ei.value.status == J.JF_ECAPACITY
        c2 = small.generate([prompts[0]], gen)  # the refused call changed nothing
        assert np.array_equal(c2.tokens, a.tokens)
    finally:
        ref.close()
        small.close()
