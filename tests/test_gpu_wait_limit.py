"""The error path of the bounded device waits (JF_ETIMEOUT), made to fire without a GPU fault.

Every wait of the kernels on a TMA copy, an MMA or the accumulator hand-over is bounded by the
context's wait limit; when one runs out the kernel records the timeout in the error word, lets its
CTA finish, and the call returns JF_ETIMEOUT. A wait that runs out beside a copy or an MMA in
flight is never provoked here. The probe waits instead, under the same limit and through the same
bounded-wait routine, on a shared-memory mbarrier that nothing arrives at: nothing is in flight
when it gives up. The tests check that the limit set on the host is the one the device honours,
that the call returns JF_ETIMEOUT and names the wait, that no kernel is left behind (the stream is
idle afterwards), and that the context then recovers: the same forward gives the same results
before and after, under the shortened limit and after the default is restored.
"""
import time

import numpy as np
import pytest

from paper_2512_14681_gb300 import inputs as I
from tests.parity import need_gpu

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def ctx():
    need_gpu()
    from paper_2512_14681_gb300.jacobi import Context

    c = Context(I.SMALL_BF16, max_seqs=1, max_ctx=512, max_rows=64, logits_rows=64)
    c.init_random_weights(I.WEIGHT_SEED, I.WEIGHT_STD)
    c.prefill(0, I.prompt_tokens(I.SMALL_BF16.vocab, 150, seed=81))
    yield c
    c.close()


def _forward(c):
    toks = I.prompt_tokens(I.SMALL_BF16.vocab, 40, seed=82)
    lg, _, am = c.forward_logits(0, toks, want_hidden=False)
    return lg.copy(), am.copy()


def test_limit_is_validated_on_the_host(ctx):
    from paper_2512_14681_gb300._lib import JF_EINVAL

    for bad in (0, 999_999, 60_000_000_001):
        assert ctx.lib.jf_set_wait_limit(ctx.h, bad) == JF_EINVAL
    assert b"wait limit" in ctx.lib.jf_last_error(ctx.h)


@pytest.mark.parametrize("limit_ms", [5, 50])
def test_probe_times_out_under_the_host_set_limit_and_the_context_recovers(ctx, limit_ms):
    import torch

    from paper_2512_14681_gb300._lib import JF_ETIMEOUT

    before = _forward(ctx)
    ctx.set_wait_limit(limit_ms * 1_000_000)
    t0 = time.perf_counter()
    status, waited_ns = ctx.wait_limit_probe()
    wall = time.perf_counter() - t0
    assert status == JF_ETIMEOUT
    assert b"timed out" in ctx.lib.jf_last_error(ctx.h)
    # the device honoured the host's limit: it gave up just after it, not after the 2 s default
    assert limit_ms * 1e6 <= waited_ns < limit_ms * 1e6 + 2e6
    assert wall < 1.0
    # nothing is left running on the device
    torch.cuda.synchronize()
    # the error word was cleared: the same forward, still under the short limit, gives the same
    # results and reports no error
    a = _forward(ctx)
    assert np.array_equal(a[0], before[0]) and np.array_equal(a[1], before[1])
    ctx.set_wait_limit(2_000_000_000)
    b = _forward(ctx)
    assert np.array_equal(b[0], before[0]) and np.array_equal(b[1], before[1])


def test_generation_after_a_timeout_matches_one_without(ctx):
    """A decode run (iteration graphs re-captured after the limit changed) after a timeout equals
    the same run before it."""
    from paper_2512_14681_gb300._lib import JF_ETIMEOUT
    from paper_2512_14681_gb300.jacobi import Gen

    prompt = I.prompt_tokens(I.SMALL_BF16.vocab, 30, seed=83)
    g = Gen(block_size=8, max_new=24)
    ctx.truncate(0, 0)
    first = ctx.generate([prompt], g)
    ctx.set_wait_limit(10_000_000)
    assert ctx.wait_limit_probe()[0] == JF_ETIMEOUT
    ctx.truncate(0, 0)
    second = ctx.generate([prompt], g)
    ctx.set_wait_limit(2_000_000_000)
    assert list(second.tokens[0]) == list(first.tokens[0])
    assert np.array_equal(second.counts, first.counts)
