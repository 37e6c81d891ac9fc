"""Forward pass of libjf vs the oracle, through the C ABI (tiny fp32 and small bf16 decoders).

* weights: both sides draw the same counter-based N(0, 0.02) stream; the device copy must equal
  the oracle's values element for element (also the Q/K/V biases, for the variants with QKV biases
  and tied embeddings);
* logits and final hidden state of one causal forward (Eq. 3) over the cache + in-flight rows:
  max-abs 1e-4 (fp32 model) / 3e-2 (bf16 model);
* the KV commit (cache trim of Algorithm 1) leaves exactly the cache a prefill of the committed
  sequence would build;
* jf_jacobi_step verifies caller-supplied RA / pseudo / candidate blocks (Algorithm 1).
"""
import numpy as np
import pytest

from oracle import oracle as O
from paper_2512_14681_gb300 import inputs as I
from tests.parity import LOGIT_TOL, need_gpu

pytestmark = pytest.mark.gpu

SHAPES = [I.TINY_F32, I.SMALL_BF16, I.TINY_F32_BT, I.SMALL_BF16_BT]


def _tids(shape, layers):
    """Tensor ids of the shape (include/jf.h): no LM head when tied, three biases a layer with
    QKV biases."""
    head = [0, 2] if shape.tie_embeddings else [0, 1, 2]
    per = 12 if shape.qkv_bias else 9
    return head + [8 + 16 * l + w for l in layers for w in range(per)]


@pytest.fixture(scope="module", params=SHAPES, ids=lambda s: s.name)
def pair(request):
    need_gpu()
    from paper_2512_14681_gb300.jacobi import Context

    shape = request.param
    ctx = Context(shape, max_seqs=2, max_ctx=512, max_rows=64, logits_rows=64)
    ctx.init_random_weights(I.WEIGHT_SEED, I.WEIGHT_STD)
    model = O.Model(O.ModelConfig(**shape.oracle_kwargs())).init_random(I.WEIGHT_SEED, I.WEIGHT_STD)
    yield shape, ctx, model
    ctx.close()


def test_weights_equal_oracle(pair):
    shape, ctx, model = pair
    tids = _tids(shape, range(shape.n_layers))
    for tid in tids:
        ref = model.get_tensor(tid)
        got = ctx.get_weights(tid, 0, ref.size).astype(np.float64)
        bad = np.nonzero(got != ref)[0]
        # the transcendental functions of the two generators may differ in the last fp64 bit,
        # which can move a value across a rounding boundary of the stored precision
        assert bad.size <= 2, f"tensor {tid}: {bad.size} mismatches"
        if bad.size:
            rel = np.abs(got[bad] - ref[bad]) / np.abs(ref[bad])
            assert rel.max() <= (2.0 ** -7 if shape.bf16 else 2.0 ** -23)


def test_forward_logits_match_oracle(pair):
    shape, ctx, model = pair
    prompt = I.prompt_tokens(shape.vocab, 48, seed=21)
    # 1) empty cache: 37 rows in flight (ragged against every tile)
    lg, hid, am = ctx.forward_logits(0, prompt[:37])
    ref = O.forward(model, O.Cache(model, 512, 64), prompt[:37], np.arange(37), want_logits=True, want_hidden=True)
    tol = LOGIT_TOL[shape.bf16]
    d = np.abs(lg - ref.logits).max()
    assert d <= tol, f"logit max-abs diff {d}"
    rel = np.abs(hid - ref.hidden).max() / np.abs(ref.hidden).max()
    assert rel <= (1e-5 if not shape.bf16 else 1e-2)
    agree = np.mean(am == ref.argmax)
    flagged = ref.margin < 2 * tol
    assert np.all((am == ref.argmax) | flagged), f"argmax disagreement outside near-ties ({agree})"
    # 2) committed cache of 29 tokens (two KV pages and a ragged one) + 11 rows in flight
    ctx.truncate(1, 0) if ctx.seq_len(1) else None
    q0 = ctx.prefill(1, prompt[:29])
    oc = O.Cache(model, 512, 64)
    pre = O.forward(model, oc, prompt[:29], np.arange(29))
    oc.commit(np.arange(29))
    assert q0 == pre.argmax[-1] or pre.margin[-1] < 2 * tol
    lg, hid, am = ctx.forward_logits(1, prompt[29:40])
    ref = O.forward(model, oc, prompt[29:40], np.arange(29, 40), want_logits=True)
    d = np.abs(lg - ref.logits).max()
    assert d <= tol, f"logit max-abs diff with cache {d}"
    ctx.truncate(1, 0)


def test_commit_equals_prefill_of_committed_sequence(pair):
    shape, ctx, model = pair
    prompt = I.prompt_tokens(shape.vocab, 40, seed=22)
    from paper_2512_14681_gb300._lib import JF_BLOCK_RA

    ctx.truncate(0, 0) if ctx.seq_len(0) else None
    q0 = ctx.prefill(0, prompt[:20])
    # a draft whose first tokens are the model's own greedy continuation, then noise
    ar = [q0]
    for _ in range(4):
        _, _, am = ctx.forward_logits(0, np.array(ar, dtype=np.int32), want_logits=False, want_hidden=False)
        ar.append(int(am[-1]))
    draft = np.array(ar[:4] + [7, 8, 9, 10], dtype=np.int32)
    out = ctx.jacobi_step(0, [(JF_BLOCK_RA, 20, 8, -1)], draft)
    k = len(out["committed"])
    assert out["counts"][0] == k and k >= 4
    assert list(out["committed"]) == list(draft[:k])
    assert ctx.seq_len(0) == 20 + k
    nxt = np.array([int(out["predictions"][k - 1])] + [11, 12], dtype=np.int32)
    a, _, _ = ctx.forward_logits(0, nxt, want_hidden=False)
    # the same sequence prefilled in one go
    ctx.truncate(1, 0) if ctx.seq_len(1) else None
    ctx.prefill(1, np.concatenate([prompt[:20], draft[:k]]))
    b, _, _ = ctx.forward_logits(1, nxt, want_hidden=False)
    assert np.abs(a - b).max() <= (1e-5 if not shape.bf16 else 2e-3)
    ctx.truncate(0, 0)
    ctx.truncate(1, 0)


def test_step_blocks_match_oracle_predictions(pair):
    """RA + pseudo block + candidate in one step; counts follow the greedy rule on the device's
    predictions and the predictions equal the oracle's (except flagged near-ties)."""
    shape, ctx, model = pair
    from paper_2512_14681_gb300._lib import JF_BLOCK_CAND, JF_BLOCK_PSEUDO, JF_BLOCK_RA

    prompt = I.prompt_tokens(shape.vocab, 30, seed=23)
    ctx.truncate(0, 0) if ctx.seq_len(0) else None
    q0 = ctx.prefill(0, prompt)
    P = 30
    ra = np.array([q0] + list(I.prompt_tokens(shape.vocab, 5, seed=24)), dtype=np.int32)
    ps = I.prompt_tokens(shape.vocab, 6, seed=25)
    cand = np.array([q0] + list(I.prompt_tokens(shape.vocab, 4, seed=26)), dtype=np.int32)
    blocks = [(JF_BLOCK_RA, P, 6, -1), (JF_BLOCK_PSEUDO, P + 6, 6, 0), (JF_BLOCK_CAND, P, 5, -1)]
    draft = np.concatenate([ra, ps, cand])
    out = ctx.jacobi_step(0, blocks, draft)
    g = out["predictions"]
    # oracle predictions with the same segments (pseudo block's parent = RA)
    oc = O.Cache(model, 512, 64)
    O.forward(model, oc, prompt, np.arange(P))
    oc.commit(np.arange(P))
    pos = np.concatenate([np.arange(P, P + 6), np.arange(P + 6, P + 12), np.arange(P, P + 5)])
    seg = np.array([0] * 6 + [1] * 6 + [2] * 5)
    ref = O.forward(model, oc, draft, pos, seg, np.array([0, 1, 0], dtype=np.uint32))
    tol = LOGIT_TOL[shape.bf16]
    assert np.all((g == ref.argmax) | (ref.margin < 2 * tol))
    # the fp32 top-2 the device reports agree with the oracle's
    assert np.abs(out["top2"][:, 0] - ref.top2[:, 0]).max() <= tol

    def lead(tokens, preds, free_first):
        k = 1 if free_first else 0
        while k < len(tokens) and tokens[k] == preds[k - 1]:
            k += 1
        return k

    k_ra = lead(ra, g[0:6], True)
    k_ps = 0
    while k_ps < 6 and ps[k_ps] == g[5 + k_ps]:
        k_ps += 1
    k_c = lead(cand, g[12:17], True)
    assert list(out["counts"]) == [k_ra, k_ps, k_c]
    k = max(k_ra, k_c)
    assert len(out["committed"]) == k
    ctx.truncate(0, 0)


def test_invalid_step_is_rejected_without_state_change(pair):
    shape, ctx, model = pair
    from paper_2512_14681_gb300._lib import JF_BLOCK_CAND, JF_BLOCK_RA, JfError

    prompt = I.prompt_tokens(shape.vocab, 10, seed=27)
    ctx.truncate(0, 0) if ctx.seq_len(0) else None
    q0 = ctx.prefill(0, prompt)
    bad = [
        ([(JF_BLOCK_RA, 11, 4, -1)], [q0, 1, 2, 3]),                      # RA not at P
        ([(JF_BLOCK_CAND, 10, 4, -1)], [q0, 1, 2, 3]),                    # no RA first
        ([(JF_BLOCK_RA, 10, 4, -1)], [q0, 1, 2, shape.vocab]),            # token out of range
        ([(JF_BLOCK_RA, 10, 65, -1)], [q0] * 65),                         # more rows than max_rows
    ]
    for blocks, draft in bad:
        with pytest.raises(JfError):
            ctx.jacobi_step(0, blocks, np.array(draft, dtype=np.int32))
        assert ctx.seq_len(0) == 10
    ctx.truncate(0, 0)


def test_weight_file_roundtrip_and_refused_files(pair, tmp_path):
    """jf_save_weights / jf_load_weights: the saved file loads back bit for bit over other weights; a
    truncated file and a file of another shape are refused with JF_EIO and leave the weights as they
    were (the whole file is read and checked before any upload)."""
    from paper_2512_14681_gb300 import _lib as J

    shape, ctx, model = pair
    tids = _tids(shape, [0])  # every tensor kind of layer 0

    def snap():
        out = {}
        for t in tids:
            n = model.get_tensor(t).size
            head = min(n, 4096)
            out[t] = np.concatenate([ctx.get_weights(t, 0, head), ctx.get_weights(t, n - head, head)])
        return out

    path = str(tmp_path / "w.jfw")
    ctx.save_weights(path)
    before = snap()
    ctx.init_random_weights(I.WEIGHT_SEED + 7, I.WEIGHT_STD)
    other = snap()
    assert any(not np.array_equal(before[t], other[t]) for t in tids if t != 2)
    ctx.load_weights(path)
    for t in tids:
        assert np.array_equal(snap()[t], before[t]), t
    data = open(path, "rb").read()
    bad = str(tmp_path / "bad.jfw")
    open(bad, "wb").write(data[: len(data) // 2])
    with pytest.raises(J.JfError) as ei:
        ctx.load_weights(bad)
    assert ei.value.status == J.JF_EIO
    wrong = bytearray(data)
    wrong[4 * 4: 4 * 4 + 4] = (int.from_bytes(data[16:20], "little") + 64).to_bytes(4, "little")  # d_model
    open(bad, "wb").write(bytes(wrong))
    with pytest.raises(J.JfError) as ei:
        ctx.load_weights(bad)
    assert ei.value.status == J.JF_EIO
    after = snap()
    for t in tids:
        assert np.array_equal(after[t], before[t]), t


def test_refused_prefill_and_truncate_leave_the_sequence(pair):
    """Host checks before any launch: a prompt past max_ctx (JF_ECAPACITY), an out-of-range token
    (JF_EINVAL), a truncate past the committed length and a bad sequence slot (JF_EINVAL)."""
    from paper_2512_14681_gb300 import _lib as J

    shape, ctx, model = pair
    ctx.truncate(0, 0) if ctx.seq_len(0) else None
    ctx.prefill(0, I.prompt_tokens(shape.vocab, 12, seed=31))
    cases = [
        (J.JF_ECAPACITY, lambda: ctx.prefill(0, I.prompt_tokens(shape.vocab, 512, seed=32))),  # 12 + 512 > 512
        (J.JF_EINVAL, lambda: ctx.prefill(0, np.array([1, shape.vocab], dtype=np.int32))),
        (J.JF_EINVAL, lambda: ctx.truncate(0, 13)),
        (J.JF_EINVAL, lambda: ctx.prefill(5, np.array([1, 2], dtype=np.int32))),               # max_seqs = 2
    ]
    for status, call in cases:
        with pytest.raises(J.JfError) as ei:
            call()
        assert ei.value.status == status
        assert ctx.seq_len(0) == 12
    ctx.truncate(0, 0)
