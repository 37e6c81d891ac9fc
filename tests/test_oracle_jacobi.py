"""Pins of the oracle's decoding loops against what the paper fixes (no GPU).

* Sec. 2.1 / Eq. 3: the Jacobi fixed point equals greedy AR decoding, and the first position of
  a block is exact each iteration, so a block of n converges in at most n iterations.
* Eq. 4: blocks compose sequentially into the AR output.
* Sec. 3.2 / Algorithm 1: multi-block decoding and rejection recycling accept tokens by greedy
  rejection sampling in the real-active block only, so they are lossless.
* Draft injection: a token at position i is accepted iff every injected token before it is
  uncorrupted, so with window n the mean accepted count is 1 + sum_{j=1}^{n-1} (1-p)^j.
"""
import math

import numpy as np
import pytest

from oracle import oracle as O
from oracle import jacobi as J
from paper_2512_14681_gb300 import inputs as I


@pytest.fixture(scope="module")
def tiny():
    return O.Model(O.ModelConfig(**I.TINY_F32.oracle_kwargs())).init_random(I.WEIGHT_SEED, I.WEIGHT_STD)


@pytest.fixture(scope="module")
def prompt():
    return I.prompt_tokens(I.TINY_F32.vocab, 32, seed=I.PROMPT_SEED)


@pytest.fixture(scope="module")
def ar64(tiny, prompt):
    return J.generate_ar(tiny, prompt, 64)


def test_ar_is_greedy_argmax_of_the_full_sequence(tiny, prompt, ar64):
    """Eq. 1 brute force: each AR token is the argmax after the full prefix, recomputed from scratch."""
    seq = list(prompt) + ar64.tokens
    for i in (0, 17, 63):
        c = O.Cache(tiny, 128, 128)
        n = len(prompt) + i
        out = O.forward(tiny, c, seq[:n], np.arange(n))
        assert out.argmax[-1] == ar64.tokens[i]


@pytest.mark.parametrize("n", [1, 3, 8, 16])
def test_block_jacobi_equals_ar_and_converges_within_n(tiny, prompt, ar64, n):
    res = J.generate_jacobi(tiny, prompt, J.GenParams(block_size=n, max_new=64))
    assert res.tokens == ar64.tokens
    assert all(it.k >= 1 for it in res.iters)
    # iterations per block <= n (block mode: a block ends when its n positions are committed)
    done, iters_in_block = 0, 0
    for it in res.iters:
        iters_in_block += 1
        done += it.k
        assert iters_in_block <= n
        if done % n == 0:
            iters_in_block = 0
    if n == 1:
        assert len(res.iters) == 64


def test_window_jacobi_equals_ar(tiny, prompt, ar64):
    res = J.generate_jacobi(tiny, prompt, J.GenParams(block_size=8, mode="window", max_new=64))
    assert res.tokens == ar64.tokens
    assert all(it.M == 8 for it in res.iters)


def test_ar_mode_is_one_token_per_forward(tiny, prompt, ar64):
    res = J.generate_jacobi(tiny, prompt, J.GenParams(mode="ar", max_new=20))
    assert res.tokens == ar64.tokens[:20] and all(it.k == 1 and it.M == 1 for it in res.iters)


@pytest.mark.parametrize("K,r", [(2, 0.0), (3, 0.5), (4, 0.0)])
def test_multiblock_is_lossless(tiny, prompt, ar64, K, r):
    res = J.generate_jacobi(tiny, prompt, J.GenParams(block_size=6, n_blocks=K, spawn_ratio=r, max_new=64))
    assert res.tokens == ar64.tokens


def test_multiblock_k1_equals_single_block(tiny, prompt):
    a = J.generate_jacobi(tiny, prompt, J.GenParams(block_size=8, max_new=40))
    b = J.generate_jacobi(tiny, prompt, J.GenParams(block_size=8, n_blocks=1, spawn_ratio=0.3, max_new=40))
    assert a.tokens == b.tokens and a.counts == b.counts and [i.M for i in a.iters] == [i.M for i in b.iters]


def test_rejection_recycling_is_lossless_and_empty_pool_is_a_no_op(tiny, prompt, ar64):
    rr = J.generate_jacobi(tiny, prompt, J.GenParams(block_size=8, pool_size=16, cand_per_iter=2, max_new=64))
    assert rr.tokens == ar64.tokens
    assert any(len(it.k_cand) > 0 for it in rr.iters)
    base = J.generate_jacobi(tiny, prompt, J.GenParams(block_size=8, max_new=64))
    off = J.generate_jacobi(tiny, prompt, J.GenParams(block_size=8, pool_size=0, cand_per_iter=2, max_new=64))
    assert off.counts == base.counts and [i.M for i in off.iters] == [i.M for i in base.iters]


def test_multiblock_with_recycling_is_lossless(tiny, prompt, ar64):
    res = J.generate_jacobi(tiny, prompt, J.GenParams(block_size=8, n_blocks=3, pool_size=8, cand_per_iter=1,
                                                      max_new=64))
    assert res.tokens == ar64.tokens


def test_recycled_candidate_wins_when_it_holds_the_continuation(tiny, prompt, ar64):
    """A pool entry keyed by q0 that carries the true continuation is accepted in full."""
    d = J.JacobiDecoder(tiny, prompt, J.GenParams(block_size=8, pool_size=4, cand_per_iter=1, max_new=64))
    d.step()
    P_new = len(d.tokens)
    ent = ar64.tokens[P_new:P_new + 8]
    assert ent[0] == d.q0
    d.pool.append(list(ent))
    Ln = len(d.blocks[0].q)
    d.cands = [([d.q0] + ent[1:])[:Ln]]
    rec = d.step()
    assert rec.winner == 1 and rec.k == Ln
    assert d.tokens == ar64.tokens[:len(d.tokens)]


def _truth(tiny, prompt, n_extra):
    return J.generate_ar(tiny, prompt, n_extra).tokens


def test_injection_extremes(tiny, prompt):
    truth = _truth(tiny, prompt, 64 + 8 + 8 + 1)
    p0 = J.generate_jacobi(tiny, prompt, J.GenParams(block_size=8, init="inject", inject_p=0.0, max_new=64), truth)
    assert p0.tokens == truth[:64]
    assert p0.counts == [8] * 8                                # whole block accepted every time
    p1 = J.generate_jacobi(tiny, prompt, J.GenParams(block_size=8, init="inject", inject_p=1.0, max_new=24), truth)
    assert p1.tokens == truth[:24] and all(k == 1 for k in p1.counts)


def test_injection_mean_count_closed_form(tiny, prompt):
    n, p, new = 8, 0.3, 600
    truth = _truth(tiny, prompt, new + n + n + 1)
    res = J.generate_jacobi(tiny, prompt, J.GenParams(block_size=n, mode="window", init="inject", inject_p=p,
                                                      seed=I.INJECT_SEED, max_new=new), truth)
    assert res.tokens == truth[:new]
    ks = np.array(res.counts[:-1], dtype=np.float64)          # last iteration may be cut by max_new
    expect = 1 + sum((1 - p) ** j for j in range(1, n))
    var = np.var(ks)
    assert abs(ks.mean() - expect) < 4.5 * math.sqrt(var / ks.size)
    assert ks.max() <= n and ks.min() >= 1


def test_injection_threshold_is_exact_for_fp32_p():
    assert J.inject_threshold(0.0) == 0
    assert J.inject_threshold(1.0) == 2**53
    assert J.inject_threshold(0.5) == 2**52
    t = J.inject_threshold(0.3)
    assert t == int(float(np.float32(0.3)) * 2**53)


def test_injected_token_differs_from_truth_when_corrupted():
    T = J.inject_threshold(1.0)
    toks = [J.inject_token(5, pos, it, 7, T, 11) for pos in range(50) for it in range(3)]
    assert all(t != 7 and 0 <= t < 11 for t in toks)
    assert len(set(toks)) == 10


def test_eos_stops_generation(tiny, prompt, ar64):
    eos = ar64.tokens[10]
    first = ar64.tokens.index(eos)
    res = J.generate_jacobi(tiny, prompt, J.GenParams(block_size=8, max_new=64, eos_id=eos))
    assert res.tokens == ar64.tokens[:first + 1]


def test_short_prompt_and_short_generation(tiny):
    p = I.prompt_tokens(I.TINY_F32.vocab, 1, seed=12)
    ar = J.generate_ar(tiny, p, 5)
    res = J.generate_jacobi(tiny, p, J.GenParams(block_size=8, max_new=5))
    assert res.tokens == ar.tokens and len(res.tokens) == 5


@pytest.mark.parametrize("init", ["repeat", "inject"])
def test_paper_inference_configuration_is_lossless(tiny, prompt, ar64, init):
    """K = 2 blocks, spawn ratio r = 0.85, 4 recycled n-grams verified per iteration (the paper's
    chosen configuration, Sec. 4.3), at a small block size: still exactly the AR greedy output."""
    # injection needs the truth beyond max_new (K n + G + 1 more tokens than are generated)
    max_new = 39 if init == "inject" else 64
    kw = dict(block_size=8, n_blocks=2, spawn_ratio=0.85, pool_size=16, cand_per_iter=4, max_new=max_new)
    if init == "inject":
        kw.update(init="inject", inject_p=0.3, seed=5)
    res = J.generate_jacobi(tiny, prompt, J.GenParams(**kw), truth=ar64.tokens if init == "inject" else None)
    assert res.tokens == ar64.tokens[:max_new]


def test_second_block_spawns_at_the_threshold(tiny, prompt, ar64):
    """Algorithm 1: the next block starts once the newest one holds ceil(r n) accepted tokens.
    With p = 0 injection every draft is exact, so the first block commits all n = 8 tokens in its
    first iteration; with r = 0.85 (threshold 7) the second block spawns right after it, never
    before. Before the spawn the forward carries only the first block's rows."""
    res = J.generate_jacobi(tiny, prompt, J.GenParams(block_size=8, n_blocks=2, spawn_ratio=0.85, init="inject",
                                                      inject_p=0.0, seed=1, max_new=32), truth=ar64.tokens)
    assert res.tokens == ar64.tokens[:32]
    assert res.iters[0].M == 8 and res.iters[0].k == 8 and res.iters[0].pseudo == []
    # a ratio of 0 (threshold 0) has both blocks in flight from the first iteration
    eager = J.generate_jacobi(tiny, prompt, J.GenParams(block_size=8, n_blocks=2, spawn_ratio=0.0, max_new=16))
    assert eager.iters[0].M == 16 and len(eager.iters[0].pseudo) == 1
