"""Jacobi trajectory collection on the device (Sec. 2.1: the trajectory J = {y^(0), ..., y^(k)} of
each block; Sec. 3.1 and App. C: the training data of Jacobi Forcing is collected from them).

jf_generate records, into a caller-lent device buffer, every row of every iteration's forward:
sequence slot, kind (real-active draft / pseudo-active block / recycled candidate), position, draft
token and greedy prediction. Checked element by element against the rows the oracle's decoding loop
builds and the predictions it takes, in several decoding modes and for a batch of two sequences. A
prediction may differ only at a flagged near-tie of the oracle (top-1/top-2 margin below twice the
logit tolerance); the comparison of that run stops at such a row.
"""
import numpy as np
import pytest

from oracle import jacobi as OJ
from oracle import oracle as O
from paper_2512_14681_gb300 import inputs as I
from tests.parity import LOGIT_TOL, need_gpu

pytestmark = pytest.mark.gpu

MODES = {
    "jacobi_block8": dict(block_size=8),
    "window6": dict(block_size=6, mode="window"),
    "mb3_r05_rr": dict(block_size=6, n_blocks=3, spawn_ratio=0.5, pool_size=8, cand_per_iter=2),
    "inj_mb2_rr_g5": dict(block_size=8, n_blocks=2, pool_size=16, cand_per_iter=1, ngram_len=5, init="inject",
                          inject_p=0.3, seed=9),
}


@pytest.fixture(scope="module", params=[I.TINY_F32, I.SMALL_BF16], ids=lambda s: s.name)
def setup(request):
    need_gpu()
    from paper_2512_14681_gb300.jacobi import Context

    shape = request.param
    ctx = Context(shape, max_seqs=2, max_ctx=512, max_rows=96)
    ctx.init_random_weights(I.WEIGHT_SEED, I.WEIGHT_STD)
    model = O.Model(O.ModelConfig(**shape.oracle_kwargs())).init_random(I.WEIGHT_SEED, I.WEIGHT_STD)
    yield shape, ctx, model
    ctx.close()


def _rows_of(rec, seq):
    mine = rec["seq"] == seq
    return {k: rec[src][mine] for k, src in (("tokens", "token"), ("pos", "pos"), ("pred", "pred"), ("kind", "kind"))}


def _compare(records, seq, ref, tol):
    """Iteration by iteration: tokens, positions and kinds exactly; predictions exactly except at a
    flagged near-tie, after which the runs may part. Returns the number of iterations compared."""
    for i, it in enumerate(ref.iters):
        got = _rows_of(records[i], seq)
        for k in ("tokens", "pos", "kind"):
            assert got[k].tolist() == list(it.rows[k]), f"iteration {i}: {k}"
        diff = np.nonzero(got["pred"] != np.array(it.rows["pred"]))[0]
        if diff.size:
            assert all(it.rows["margin"][r] < 2 * tol for r in diff), f"iteration {i}: predictions differ at {diff}"
            return i + 1
    return len(ref.iters)


@pytest.mark.parametrize("mode", list(MODES))
def test_trajectory_matches_oracle(setup, mode):
    torch = need_gpu()
    shape, ctx, model = setup
    from paper_2512_14681_gb300.jacobi import Gen, trajectory_records

    kw = MODES[mode]
    prompt = I.prompt_tokens(shape.vocab, 29, seed=61)
    truth = None
    if kw.get("init") == "inject":
        truth = OJ.generate_ar(model, prompt, 40 + 2 * 8 + 8 + 1).tokens
    ref = OJ.generate_jacobi(model, prompt, OJ.GenParams(max_new=40, **kw), truth=truth)
    R, cap = 96, 128
    buf = torch.full((cap * (2 + 5 * R),), -5, dtype=torch.int32, device="cuda")
    tr = None if truth is None else np.array([truth], dtype=np.int32)
    out = ctx.generate([prompt], Gen(max_new=40, **kw), truth=tr, traj=buf, traj_rows=R)
    assert out.traj_iters == out.iterations
    recs = trajectory_records(buf, out.traj_iters, R)
    assert [r["it"] for r in recs] == list(range(out.iterations))
    assert [r["M"] for r in recs] == out.rows.tolist()
    n = _compare(recs, 0, ref, LOGIT_TOL[shape.bf16])
    assert n >= 1
    # recording changes nothing in the decoding itself
    plain = ctx.generate([prompt], Gen(max_new=40, **kw), truth=tr)
    assert np.array_equal(plain.tokens, out.tokens) and np.array_equal(plain.counts, out.counts)


def test_trajectory_of_a_batch(setup):
    """Two sequences decode in lockstep: each row carries its slot, and each sequence's rows are the
    rows of its own oracle run."""
    torch = need_gpu()
    shape, ctx, model = setup
    from paper_2512_14681_gb300.jacobi import Gen, trajectory_records

    kw = dict(block_size=8, n_blocks=2, pool_size=8, cand_per_iter=1)
    prompts = [I.prompt_tokens(shape.vocab, L, seed=70 + L) for L in (23, 9)]
    R, cap = 96, 64
    buf = torch.zeros(cap * (2 + 5 * R), dtype=torch.int32, device="cuda")
    out = ctx.generate(prompts, Gen(max_new=24, **kw), traj=buf, traj_rows=R)
    recs = trajectory_records(buf, out.traj_iters, R)
    for r in recs:
        assert set(np.unique(r["seq"]).tolist()) <= {0, 1}
    for b, p in enumerate(prompts):
        ref = OJ.generate_jacobi(model, p, OJ.GenParams(max_new=24, **kw))
        assert _compare(recs, b, ref, LOGIT_TOL[shape.bf16]) >= 1


def test_trajectory_buffer_is_checked(setup):
    """A buffer with fewer rows than one forward is refused before any launch; a buffer with fewer
    iterations than the decoding records the first ones only."""
    torch = need_gpu()
    shape, ctx, model = setup
    from paper_2512_14681_gb300 import _lib as J
    from paper_2512_14681_gb300.jacobi import Gen, trajectory_records

    prompt = I.prompt_tokens(shape.vocab, 12, seed=62)
    small = torch.zeros(4 * (2 + 5 * 7), dtype=torch.int32, device="cuda")
    with pytest.raises(J.JfError) as ei:
        ctx.generate([prompt], Gen(block_size=8, max_new=8), traj=small, traj_rows=7)
    assert ei.value.status == J.JF_EINVAL
    R = 8
    buf = torch.full((3 * (2 + 5 * R) + 5,), -5, dtype=torch.int32, device="cuda")
    out = ctx.generate([prompt], Gen(block_size=8, max_new=20), traj=buf, traj_rows=R)
    assert out.iterations > 3 and out.traj_iters == 3
    recs = trajectory_records(buf, 3, R)
    assert [r["it"] for r in recs] == [0, 1, 2]
    assert buf[-5:].tolist() == [-5] * 5  # nothing written past the last record


@pytest.mark.parametrize("n,w", [(8, 2), (8, 4), (4, 8)])
def test_training_points_match_oracle(setup, n, w):
    """App. C with Eq. 2's schedule (jf_trajectory_noisy_blocks): the point each block's trajectory
    contributes as its noisy training block, picked on the device from the device's trajectory record,
    equals the oracle's pick from its own decoding loop (blocks whose trajectories agree)."""
    torch = need_gpu()
    shape, ctx, model = setup
    from paper_2512_14681_gb300.jacobi import Gen, trajectory_noisy_blocks, trajectory_records

    prompt = I.prompt_tokens(shape.vocab, 21, seed=63)
    max_new = 40
    ref = OJ.generate_jacobi(model, prompt, OJ.GenParams(block_size=n, max_new=max_new))
    R, cap = 16, 256
    buf = torch.zeros(cap * (2 + 5 * R), dtype=torch.int32, device="cuda")
    out = ctx.generate([prompt], Gen(block_size=n, max_new=max_new), traj=buf, traj_rows=R)
    recs = trajectory_records(buf, out.traj_iters, R)
    same = _compare(recs, 0, ref, LOGIT_TOL[shape.bf16])  # iterations whose rows and predictions agree
    new = torch.from_numpy(out.tokens[0].astype(np.int32)).cuda()
    noisy, point = trajectory_noisy_blocks(buf, out.traj_iters, R, 0, new, prompt.size, n, w)
    noisy, point = noisy.cpu().numpy(), point.cpu().numpy()
    picks = OJ.noisy_blocks(ref, prompt.size, n, w)
    assert len(picks) == max_new // n == point.size
    checked = 0
    for i, (j, toks) in enumerate(picks):
        pts = [p for p, _ in OJ.block_points(ref, prompt.size, n, i)[:-1]]
        if pts and max(pts) >= same:
            break  # from here the two runs may have parted at a near-tie
        got_j = int(point[i])
        assert (got_j if got_j < out.traj_iters else len(ref.iters)) == j, f"block {i}"
        assert noisy[i].tolist() == list(toks), f"block {i}"
        checked += 1
    assert checked >= 1
