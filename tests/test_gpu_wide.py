"""Element-wise oracle parity of wide forwards: the 7B per-layer widths and many rows in flight.

One Jacobi iteration is one causal forward over every in-flight row (Sec. 2.1, Eq. 3); with
multi-block decoding and rejection recycling (Sec. 3.2, Algorithm 1) those rows are the real-active
draft, the pseudo-active blocks after it and the recycled candidates beside it. These tests compare
the device with the oracle, element by element, at the row counts and widths the decode workloads
run:
* a two-layer copy of the Qwen2.5-7B shape (d 3584, 28/4 heads, MLP 18944, vocabulary 152064 --
  every per-layer width of the 7B model) over a committed cache of 1,100 tokens: fp32 logits of a
  32-row forward, and the predictions and top-2 logits of 160-row (real-active + 3 pseudo blocks + 1
  candidate, n = 32) and 384-row (the paper's K = 2, n = 64 configuration with 4 candidates) steps;
* the tiny fp32 and small bf16 shapes at 128, 160, 256 and 300 rows, so that every token-tile width
  of the projections (128, 160, 256 and two 256-row tiles) and several query tiles per attention
  unit run end to end.
Logits: max-abs 1e-4 (fp32 model) / 3e-2 (bf16 model); at the 7B widths the bf16 bound is twice the
spread that one fp32 unit at every bf16 rounding point gives the oracle's own logits, when that is
larger (tests/golden/logit_noise_floor.json). Greedy decisions equal outside the oracle's near-ties
(top-1/top-2 margin below twice the tolerance).
"""
import numpy as np
import pytest

from oracle import oracle as O
from paper_2512_14681_gb300 import inputs as I
from tests.parity import LOGIT_TOL, need_gpu, wide_logit_tol

pytestmark = pytest.mark.gpu

P_WIDE = 1100          # committed tokens under the 7B-width steps (69 pages, the last one ragged)
PREFILL_CHUNK = 384    # rows of one prefill forward, on both sides


def _oracle_prefill(model, oc, prompt, chunk):
    for s in range(0, prompt.size, chunk):
        e = min(prompt.size, s + chunk)
        out = O.forward(model, oc, prompt[s:e], np.arange(s, e))
        oc.commit(np.arange(e - s))
    return out


def _check_step(ctx, model, oc, P, blocks, draft, tol):
    """One jf_jacobi_step against the oracle's forward with the same segments: predictions outside
    near-ties, both top-2 logits, and the counts / committed tokens that follow from the device's
    own predictions under the acceptance rule. Leaves the sequence at length P again."""
    from paper_2512_14681_gb300._lib import JF_BLOCK_CAND, JF_BLOCK_PSEUDO, JF_BLOCK_RA

    out = ctx.jacobi_step(0, blocks, draft)
    g = out["predictions"]
    pos, seg, anc = [], [], []
    for b, (kind, start, n, parent) in enumerate(blocks):
        pos += list(range(start, start + n))
        seg += [b] * n
        # a pseudo block sees its parent chain; the real-active block and candidates see only the cache
        anc.append(anc[parent] | (1 << parent) if kind == JF_BLOCK_PSEUDO else 0)
    ref = O.forward(model, oc, draft, np.array(pos), np.array(seg), np.array(anc, dtype=np.uint32))
    flagged = ref.margin < 2 * tol
    bad = np.nonzero((g != ref.argmax) & ~flagged)[0]
    assert bad.size == 0, f"predictions differ from the oracle at rows {bad[:10]}"
    d = np.abs(out["top2"] - ref.top2).max()
    assert d <= tol, f"top-2 logits max-abs diff {d}"
    counts, r0, best, best_k = [], 0, 0, -1
    for b, (kind, start, n, parent) in enumerate(blocks):
        t = draft[r0:r0 + n]
        if kind == JF_BLOCK_PSEUDO:
            prev = r0 - 1  # the row before a pseudo block is the last row of its parent
            k = 0
            while k < n and t[k] == g[prev + k]:
                k += 1
        else:
            k = 1
            while k < n and t[k] == g[r0 + k - 1]:
                k += 1
            if kind in (JF_BLOCK_RA, JF_BLOCK_CAND) and k > best_k:
                best, best_k = r0, k
        counts.append(k)
        r0 += n
    assert list(out["counts"]) == counts
    assert list(out["committed"]) == list(draft[best:best + best_k])
    assert ctx.seq_len(0) == P + best_k
    ctx.truncate(0, P)
    return int(flagged.sum())


def _blocks(P, ra, n_pseudo, n_cand, n):
    from paper_2512_14681_gb300._lib import JF_BLOCK_CAND, JF_BLOCK_PSEUDO, JF_BLOCK_RA

    bl = [(JF_BLOCK_RA, P, ra, -1)]
    for j in range(n_pseudo):
        bl.append((JF_BLOCK_PSEUDO, P + ra + j * n, n, j))
    bl += [(JF_BLOCK_CAND, P, n, -1)] * n_cand
    return bl


def _draft(vocab, q0, blocks, seed, share=None):
    """Draft tokens: every real-active / candidate block starts with q0; candidate c copies the
    first `share[c]` tokens of the real-active draft so that acceptance runs differ per block."""
    rng = np.random.default_rng(seed)
    parts, ra = [], None
    for b, (kind, start, n, parent) in enumerate(blocks):
        t = rng.integers(0, vocab, size=n).astype(np.int32)
        if kind != 1:
            t[0] = q0
        if kind == 0:
            ra = t
        elif kind == 2 and share:
            k = share.pop(0)
            t[:k] = ra[:k]
        parts.append(t)
    return np.concatenate(parts).astype(np.int32)


# ---------------------------------------------------------------------------------------------
# 7B widths (two layers), 1,100-token cache
# ---------------------------------------------------------------------------------------------
@pytest.fixture(scope="module")
def wide():
    torch = need_gpu()
    from paper_2512_14681_gb300.jacobi import Context

    shape = I.QWEN7B_2L_BF16
    free, _ = torch.cuda.mem_get_info()
    if free < shape.weight_bytes() * 1.5:
        pytest.skip("not enough device memory")
    ctx = Context(shape, max_seqs=2, max_ctx=2048, max_rows=PREFILL_CHUNK, logits_rows=32)
    ctx.init_random_weights(I.WEIGHT_SEED, I.WEIGHT_STD)
    model = O.Model(O.ModelConfig(**shape.oracle_kwargs())).init_random(I.WEIGHT_SEED, I.WEIGHT_STD)
    prompt = I.prompt_tokens(shape.vocab, P_WIDE, seed=51)
    q0 = ctx.prefill(0, prompt)
    oc = O.Cache(model, 2048, PREFILL_CHUNK)
    last = _oracle_prefill(model, oc, prompt, PREFILL_CHUNK)
    tol = LOGIT_TOL[True]
    assert q0 == last.argmax[-1] or last.margin[-1] < 2 * tol
    yield shape, ctx, model, oc, int(last.argmax[-1])
    ctx.close()


def test_wide_forward_logits_32_rows(wide):
    shape, ctx, model, oc, q0 = wide
    rows = np.concatenate([[q0], I.prompt_tokens(shape.vocab, 31, seed=52)]).astype(np.int32)
    lg, hid, am = ctx.forward_logits(0, rows)
    assert ctx.seq_len(0) == P_WIDE
    ref = O.forward(model, oc, rows, np.arange(P_WIDE, P_WIDE + 32), want_logits=True, want_hidden=True)
    # at the 7B widths one fp32 unit at every bf16 rounding point already moves the oracle's own logits
    # by about 3e-2 (tests/golden/logit_noise_floor.json): the bound is twice that spread
    tol, sd_tol = wide_logit_tol("wide-7b-2layer-32rows")
    diff = np.abs(lg - ref.logits)
    assert diff.max() <= tol, f"logit max-abs diff {diff.max()} (bound {tol})"
    assert diff.std() <= sd_tol, f"logit diff std {diff.std()} (bound {sd_tol})"
    assert np.all((am == ref.argmax) | (ref.margin < 2 * tol))


def test_wide_step_160_rows(wide):
    """Real-active block + 3 pseudo blocks + 1 candidate of n = 32 (the multi-block workload)."""
    shape, ctx, model, oc, q0 = wide
    blocks = _blocks(P_WIDE, 32, 3, 1, 32)
    draft = _draft(shape.vocab, q0, blocks, seed=53, share=[5])
    assert draft.size == 160
    _check_step(ctx, model, oc, P_WIDE, blocks, draft, LOGIT_TOL[True])


def test_wide_step_384_rows(wide):
    """The paper's inference configuration: K = 2 blocks of n = 64 and 4 verified candidates."""
    shape, ctx, model, oc, q0 = wide
    blocks = _blocks(P_WIDE, 64, 1, 4, 64)
    draft = _draft(shape.vocab, q0, blocks, seed=54, share=[1, 3, 9, 2])
    assert draft.size == 384
    _check_step(ctx, model, oc, P_WIDE, blocks, draft, LOGIT_TOL[True])


# ---------------------------------------------------------------------------------------------
# many rows on the tiny fp32 and small bf16 shapes
# ---------------------------------------------------------------------------------------------
@pytest.fixture(scope="module", params=[I.TINY_F32, I.SMALL_BF16], ids=lambda s: s.name)
def many(request):
    need_gpu()
    from paper_2512_14681_gb300.jacobi import Context

    shape = request.param
    ctx = Context(shape, max_seqs=2, max_ctx=1024, max_rows=320, logits_rows=320)
    ctx.init_random_weights(I.WEIGHT_SEED, I.WEIGHT_STD)
    model = O.Model(O.ModelConfig(**shape.oracle_kwargs())).init_random(I.WEIGHT_SEED, I.WEIGHT_STD)
    prompt = I.prompt_tokens(shape.vocab, 203, seed=55)
    ctx.prefill(0, prompt)
    oc = O.Cache(model, 1024, 320)
    last = _oracle_prefill(model, oc, prompt, 320)
    yield shape, ctx, model, oc, int(last.argmax[-1])
    ctx.close()


@pytest.mark.parametrize("rows", [128, 160, 256, 300])
def test_many_rows_forward_logits(many, rows):
    shape, ctx, model, oc, q0 = many
    P = 203
    toks = I.prompt_tokens(shape.vocab, rows, seed=56 + rows)
    lg, _, am = ctx.forward_logits(0, toks, want_hidden=False)
    ref = O.forward(model, oc, toks, np.arange(P, P + rows), want_logits=True)
    tol = LOGIT_TOL[shape.bf16]
    d = np.abs(lg - ref.logits).max()
    assert d <= tol, f"{rows} rows: logit max-abs diff {d}"
    assert np.all((am == ref.argmax) | (ref.margin < 2 * tol))


@pytest.mark.parametrize("layout", ["160:ra40+2x40+cand40", "300:ra60+2x60+2cand60"])
def test_many_rows_step(many, layout):
    shape, ctx, model, oc, q0 = many
    P = 203
    if layout.startswith("160"):
        blocks = _blocks(P, 40, 2, 1, 40)
        share = [7]
    else:
        blocks = _blocks(P, 60, 2, 2, 60)
        share = [2, 11]
    draft = _draft(shape.vocab, q0, blocks, seed=57, share=share)
    assert draft.size == int(layout.split(":")[0])
    _check_step(ctx, model, oc, P, blocks, draft, LOGIT_TOL[shape.bf16])
