"""Pins of the CPU oracle against what the paper and the mathematics fix (no GPU).

Each test checks the oracle against something other than itself: a published reference
vector, a closed form, a library routine, an invariant, or brute force on tiny inputs.
Jacobi Forcing (arXiv 2512.14681) fixes: greedy Jacobi decoding reaches the greedy AR result
(Sec. 2.1, Eq. 3 and the cited proof), one causal forward solves all n conditionals (Eq. 3),
blocks compose sequentially (Eq. 4), multi-block decoding and rejection recycling are lossless
(Sec. 3.2), and the first position of a Jacobi block is exact every iteration (Eq. 3).
"""
import math

import numpy as np
import pytest

from oracle import oracle as O
from oracle import jacobi as J
from paper_2512_14681_gb300 import inputs as I


# ------------------------------------------------------------------------------------------
# Random numbers
# ------------------------------------------------------------------------------------------
def test_splitmix64_published_vector():
    # Reference outputs of SplitMix64 started at state 0 (Vigna's splitmix64.c).
    assert O.sm64(0, 0) == 0xE220A8397B1DCDAF
    assert O.sm64(0, 1) == 0x6E789E6AA1B965F4
    assert O.sm64(0, 2) == 0x06C45D188009454F


def test_normal_moments():
    z = np.array([O.normal(7, 3, e) for e in range(120000)])
    assert abs(z.mean()) < 0.015
    assert abs(z.std() - 1.0) < 0.01
    kurt = np.mean((z - z.mean()) ** 4) / z.var() ** 2
    assert abs(kurt - 3.0) < 0.08
    assert abs(np.mean(np.abs(z) < 1.0) - 0.682689) < 0.006
    # even and odd members of a pair are uncorrelated
    assert abs(np.corrcoef(z[0::2], z[1::2])[0, 1]) < 0.015


def test_weights_follow_n_0_002_and_streams_differ():
    m = O.Model(O.ModelConfig(**I.TINY_F32.oracle_kwargs())).init_random(0, 0.02)
    w = m.get_tensor(O.layer_tid(0, O.L_WG))
    assert abs(w.std() - 0.02) < 4e-4 and abs(w.mean()) < 3e-4
    w2 = m.get_tensor(O.layer_tid(0, O.L_WU))
    assert not np.allclose(w[:1000], w2[:1000])
    # gains are 1.0
    assert np.all(m.get_tensor(O.layer_tid(1, O.L_MNORM)) == 1.0)


# ------------------------------------------------------------------------------------------
# bf16 rounding
# ------------------------------------------------------------------------------------------
def test_bf16_round_ties_to_even():
    assert O.round_bf16(1.0) == 1.0
    assert O.round_bf16(1 + 2**-8) == 1.0                      # tie -> even mantissa 0
    assert O.round_bf16(1 + 3 * 2**-8) == 1 + 2**-6            # tie -> even mantissa 2
    assert O.round_bf16(1 + 2**-8 + 2**-20) == 1 + 2**-7       # above the tie
    assert O.round_bf16(-(1 + 3 * 2**-8)) == -(1 + 2**-6)
    assert O.round_bf16(0.0) == 0.0


def test_bf16_round_matches_torch():
    torch = pytest.importorskip("torch")
    x = I.random_array(4000, seed=5, scale=3.0).astype(np.float32)
    x[:10] = np.array([1e-30, -1e-38, 3e38, 65504.0, 1.00390625, 2.0**-126, 5e-39, 1.5, -7.25, 0.1], dtype=np.float32)
    ref = torch.from_numpy(x).to(torch.bfloat16).to(torch.float64).numpy()
    ours = np.array([O.round_bf16(float(v)) for v in x])
    assert np.array_equal(ours, ref)


# ------------------------------------------------------------------------------------------
# Building blocks
# ------------------------------------------------------------------------------------------
def test_rmsnorm_closed_form():
    y = O.rmsnorm([3.0, 4.0], [1.0, 1.0], 0.0)
    r = math.sqrt((9 + 16) / 2)
    assert np.allclose(y, [3 / r, 4 / r], rtol=0, atol=1e-15)
    x = I.random_array(64, seed=1).astype(np.float64)
    g = I.random_array(64, seed=2).astype(np.float64)
    assert np.allclose(O.rmsnorm(5.0 * x, g, 0.0), O.rmsnorm(x, g, 0.0), atol=1e-14)
    assert np.allclose(O.rmsnorm(x, g, 0.0), O.rmsnorm(x, np.ones(64), 0.0) * g, atol=1e-14)
    y = O.rmsnorm(x, np.ones(64), 0.0)
    assert abs(np.mean(y * y) - 1.0) < 1e-13
    assert np.all(O.rmsnorm(np.zeros(8), np.ones(8), 1e-6) == 0.0)


def test_rope_closed_forms():
    # hd = 2: one pair with frequency theta^0 = 1, so position p rotates by p radians
    assert np.allclose(O.rope([1.0, 0.0], 3, 1e4), [math.cos(3), math.sin(3)], atol=1e-15)
    # hd = 4, theta = 100: pair (1, 3) has frequency 100^(-2/4) = 0.1
    assert np.allclose(O.rope([0.0, 1.0, 0.0, 0.0], 5, 100.0), [0, math.cos(0.5), 0, math.sin(0.5)], atol=1e-15)
    v = I.random_array(128, seed=3).astype(np.float64)
    assert np.array_equal(O.rope(v, 0, 1e6), v)                # position 0 is the identity
    r = O.rope(v, 777, 1e6)
    assert np.allclose(r[:64] ** 2 + r[64:] ** 2, v[:64] ** 2 + v[64:] ** 2, atol=1e-12)
    # scores depend on relative position only
    q = I.random_array(128, seed=4).astype(np.float64)
    a = np.dot(O.rope(q, 50, 1e4), O.rope(v, 20, 1e4))
    b = np.dot(O.rope(q, 1030, 1e4), O.rope(v, 1000, 1e4))
    assert abs(a - b) < 1e-9


def test_silu_closed_forms():
    assert O.silu(0.0) == 0.0
    assert abs(O.silu(1.0) - 1.0 / (1.0 + math.exp(-1.0))) < 1e-15
    for x in (-3.0, -0.5, 0.25, 2.0, 9.0):
        assert abs((O.silu(x) - O.silu(-x)) - x) < 1e-14       # x s(x) + x s(-x) = x
    assert abs(O.silu(-40.0)) < 1e-15 and abs(O.silu(40.0) - 40.0) < 1e-12


def test_linear_matches_numpy():
    x = I.random_array((5, 33), seed=6).astype(np.float64)
    W = I.random_array((17, 33), seed=7).astype(np.float64)
    assert np.allclose(O.linear(x, W), x @ W.T, rtol=1e-13, atol=1e-13)


def test_attention_uniform_when_query_is_zero():
    Hq, Hkv, hd, n = 4, 2, 8, 7
    k = I.random_array((n, Hkv, hd), seed=8).astype(np.float64)
    v = I.random_array((n, Hkv, hd), seed=9).astype(np.float64)
    vis = np.array([1, 0, 1, 1, 0, 1, 1], dtype=np.uint8)
    out = O.attend(np.zeros((Hq, hd)), k, v, vis, Hkv)
    for h in range(Hq):
        kvh = h // (Hq // Hkv)                                  # GQA: head h reads KV head h // group
        assert np.allclose(out[h], v[vis == 1, kvh].mean(axis=0), atol=1e-14)


def test_attention_two_key_closed_form():
    hd, a = 4, 1.7
    q = np.array([[a, 0, 0, 0]], dtype=np.float64)
    k = np.zeros((2, 1, hd))
    k[0, 0, 0] = 1.0
    v = np.zeros((2, 1, hd))
    v[0, 0, 1] = 1.0
    v[1, 0, 2] = 1.0
    out = O.attend(q, k, v, np.array([1, 1], np.uint8), 1)
    w1 = math.exp(a / 2) / (math.exp(a / 2) + 1.0)              # scores a/sqrt(4) and 0
    assert np.allclose(out[0], [0, w1, 1 - w1, 0], atol=1e-15)


def test_attention_masked_keys_do_not_matter_and_empty_gives_zero():
    Hq, Hkv, hd, n = 2, 1, 8, 5
    q = I.random_array((Hq, hd), seed=10).astype(np.float64)
    k = I.random_array((n, Hkv, hd), seed=11).astype(np.float64)
    v = I.random_array((n, Hkv, hd), seed=12).astype(np.float64)
    vis = np.array([1, 1, 0, 1, 0], np.uint8)
    out = O.attend(q, k, v, vis, Hkv)
    k2, v2 = k.copy(), v.copy()
    k2[[2, 4]] += 5.0
    v2[[2, 4]] -= 3.0
    assert np.array_equal(out, O.attend(q, k2, v2, vis, Hkv))
    assert np.all(O.attend(q, k, v, np.zeros(n, np.uint8), Hkv) == 0.0)


def test_argmax_lowest_id_on_ties_and_top2():
    x = np.array([0.5, 2.0, -1.0, 2.0, 1.9])
    a, t2 = O.argmax_f32(x)
    assert a == 1 and t2[0] == np.float32(2.0) and t2[1] == np.float32(2.0)
    a, t2 = O.argmax_f32(np.array([3.0, 1.0, 2.5]))
    assert a == 0 and t2[1] == np.float32(2.5)
    # decided in fp32: values equal after rounding to fp32 tie
    a, _ = O.argmax_f32(np.array([1.0, 1.0 + 1e-12]))
    assert a == 0


# ------------------------------------------------------------------------------------------
# Whole model
# ------------------------------------------------------------------------------------------
def _tiny(seed=0, bf16=False, layers=2):
    kw = I.TINY_F32.oracle_kwargs()
    kw.update(bf16=bf16, n_layers=layers)
    return O.Model(O.ModelConfig(**kw)).init_random(seed, 0.02)


def test_one_causal_forward_equals_incremental_forwards():
    """Eq. 3: a causal forward over n rows gives the n conditionals of n separate steps."""
    m = _tiny()
    toks = I.prompt_tokens(4096, 12, seed=3)
    c1 = O.Cache(m, 64, 16)
    full = O.forward(m, c1, toks, np.arange(12), want_logits=True)
    c2 = O.Cache(m, 64, 16)
    for i in range(12):
        o = O.forward(m, c2, toks[i:i + 1], [i], want_logits=True)
        c2.commit([0])
        assert np.allclose(o.logits[0], full.logits[i], rtol=0, atol=1e-12)
        assert o.argmax[0] == full.argmax[i]


def test_tree_mask_segments():
    """A candidate segment (no ancestor) sees only the cache and itself; a child segment sees
    its ancestor's keys and itself causally, i.e. the same as one causal sequence."""
    m = _tiny()
    prompt = I.prompt_tokens(4096, 9, seed=4)
    a = I.prompt_tokens(4096, 5, seed=5)
    b = I.prompt_tokens(4096, 4, seed=6)
    cand = I.prompt_tokens(4096, 5, seed=7)

    def fresh():
        c = O.Cache(m, 64, 32)
        O.forward(m, c, prompt, np.arange(9))
        c.commit(np.arange(9))
        return c

    P = 9
    toks = np.concatenate([a, b, cand])
    pos = np.concatenate([np.arange(P, P + 5), np.arange(P + 5, P + 9), np.arange(P, P + 5)])
    seg = np.array([0] * 5 + [1] * 4 + [2] * 5)
    anc = np.array([0, 1, 0], dtype=np.uint32)
    tree = O.forward(m, fresh(), toks, pos, seg, anc, want_logits=True)
    chain = O.forward(m, fresh(), np.concatenate([a, b]), np.arange(P, P + 9), want_logits=True)
    alone = O.forward(m, fresh(), cand, np.arange(P, P + 5), want_logits=True)
    assert np.allclose(tree.logits[:9], chain.logits, atol=1e-12)
    assert np.allclose(tree.logits[9:], alone.logits, atol=1e-12)


def test_zero_layers_reduce_to_norm_and_lm_head():
    m = _tiny()
    cfg = m.cfg
    for l in range(cfg.n_layers):
        for w in (O.L_WO, O.L_WD):
            r, k = m.shape(O.layer_tid(l, w))
            m.set_tensor(O.layer_tid(l, w), np.zeros(r * k))
    E = m.get_tensor(O.T_EMBED).reshape(cfg.vocab, cfg.d_model)
    W = m.get_tensor(O.T_LMHEAD).reshape(cfg.vocab, cfg.d_model)
    toks = I.prompt_tokens(cfg.vocab, 6, seed=8)
    out = O.forward(m, O.Cache(m, 16, 8), toks, np.arange(6), want_logits=True)
    x = E[toks]
    h = x / np.sqrt(np.mean(x * x, axis=1, keepdims=True) + cfg.rms_eps)
    assert np.allclose(out.logits, h @ W.T, atol=1e-12)
    assert np.array_equal(out.argmax, np.argmax((h @ W.T).astype(np.float32), axis=1))


def test_attention_block_with_zero_queries_is_causal_mean():
    """One layer, Wq = 0 (uniform attention), Wv = [I 0], Wo = I, no MLP: row i adds the mean
    over j <= i of the normalised inputs' first hd features, to both query heads (GQA)."""
    cfg = O.ModelConfig(n_layers=1, d_model=8, n_heads=2, n_kv_heads=1, head_dim=4, d_ff=4, vocab=32)
    m = O.Model(cfg).init_random(3, 0.5)
    m.set_tensor(O.layer_tid(0, O.L_WQ), np.zeros(8 * 8))
    m.set_tensor(O.layer_tid(0, O.L_WV), np.hstack([np.eye(4), np.zeros((4, 4))]))
    m.set_tensor(O.layer_tid(0, O.L_WO), np.eye(8))
    m.set_tensor(O.layer_tid(0, O.L_WD), np.zeros(8 * 4))
    toks = np.array([3, 17, 5, 5, 30], dtype=np.int32)
    out = O.forward(m, O.Cache(m, 8, 8), toks, np.arange(5), want_hidden=True)
    E = m.get_tensor(O.T_EMBED).reshape(32, 8)
    x = E[toks]
    h = x / np.sqrt(np.mean(x * x, axis=1, keepdims=True) + cfg.rms_eps)
    for i in range(5):
        mean = h[: i + 1, :4].mean(axis=0)
        assert np.allclose(out.hidden[i], x[i] + np.concatenate([mean, mean]), atol=1e-13)


def test_mlp_block_closed_form():
    """One layer, attention output zero, W_gate = I, W_up = 2 I, W_down = 3 I: x + 3 silu(h) (2 h).
    The gate and up scales differ, so SiLU applied to the wrong branch is caught."""
    cfg = O.ModelConfig(n_layers=1, d_model=6, n_heads=2, n_kv_heads=2, head_dim=2, d_ff=6, vocab=16)
    m = O.Model(cfg).init_random(4, 0.5)
    r, k = m.shape(O.layer_tid(0, O.L_WO))
    m.set_tensor(O.layer_tid(0, O.L_WO), np.zeros(r * k))
    for w, sc in ((O.L_WG, 1.0), (O.L_WU, 2.0), (O.L_WD, 3.0)):
        m.set_tensor(O.layer_tid(0, w), sc * np.eye(6))
    toks = np.array([1, 9, 4], dtype=np.int32)
    out = O.forward(m, O.Cache(m, 8, 8), toks, np.arange(3), want_hidden=True)
    x = m.get_tensor(O.T_EMBED).reshape(16, 6)[toks]
    h = x / np.sqrt(np.mean(x * x, axis=1, keepdims=True) + cfg.rms_eps)
    assert np.allclose(out.hidden, x + 3.0 * (h / (1 + np.exp(-h))) * (2.0 * h), atol=1e-13)


def test_positions_enter_through_relative_rotation():
    """Shifting every position leaves logits unchanged (relative encoding) while swapping two
    earlier tokens changes the last row (order matters, so rotation is applied)."""
    m = _tiny()
    toks = I.prompt_tokens(4096, 7, seed=9)
    a = O.forward(m, O.Cache(m, 512, 8), toks, np.arange(7), want_logits=True)
    b = O.forward(m, O.Cache(m, 512, 8), toks, np.arange(300, 307), want_logits=True)
    assert np.allclose(a.logits, b.logits, atol=1e-9)
    sw = toks.copy()
    sw[[1, 3]] = sw[[3, 1]]
    c = O.forward(m, O.Cache(m, 512, 8), sw, np.arange(7), want_logits=True)
    assert np.max(np.abs(c.logits[-1] - a.logits[-1])) > 1e-6


def test_commit_copies_selected_rows_in_order():
    m = _tiny()
    c = O.Cache(m, 32, 8)
    toks = I.prompt_tokens(4096, 4, seed=10)
    O.forward(m, c, toks, [0, 1, 2, 3])
    c2 = O.Cache(m, 32, 8)
    O.forward(m, c2, toks[:1], [0])
    c2.commit([0])
    c.commit([0])
    assert np.array_equal(c.entry(1, 0, 0), c2.entry(1, 0, 0))
    assert np.array_equal(c.entry(0, 1, 0), c2.entry(0, 1, 0))
    with pytest.raises(ValueError):
        c.truncate(5)
    c.truncate(0)
    assert len(c) == 0


def test_bf16_model_is_close_to_fp32_model():
    """The bf16 model differs from the same weights in fp32 only by bf16 rounding."""
    m32 = _tiny(bf16=False)
    m16 = _tiny(bf16=True)
    w32 = m32.get_tensor(O.layer_tid(0, O.L_WQ))
    w16 = m16.get_tensor(O.layer_tid(0, O.L_WQ))
    assert np.array_equal(w16, np.array([O.round_bf16(v) for v in w32]))
    toks = I.prompt_tokens(4096, 8, seed=11)
    a = O.forward(m32, O.Cache(m32, 16, 8), toks, np.arange(8), want_logits=True)
    b = O.forward(m16, O.Cache(m16, 16, 8), toks, np.arange(8), want_logits=True)
    assert np.max(np.abs(a.logits - b.logits)) < 0.05


def _bf(a):
    """bf16 rounding (nearest, ties to even) by PyTorch, independent of the oracle's own routine."""
    torch = pytest.importorskip("torch")
    return torch.tensor(np.asarray(a, dtype=np.float64)).to(torch.bfloat16).to(torch.float64).numpy()


def _bf16_layer_model(d, Hq, Hkv, hd, F, V):
    cfg = O.ModelConfig(n_layers=1, d_model=d, n_heads=Hq, n_kv_heads=Hkv, head_dim=hd, d_ff=F, vocab=V, bf16=True)
    return cfg, O.Model(cfg).init_random(6, 0.5)


def test_bf16_final_norm_output_is_rounded():
    """bf16 model, no layer contribution (W_o = W_down = 0), LM head = I: the logits are the final
    RMSNorm output rounded to bf16, the precision the LM-head product takes its input in."""
    cfg, m = _bf16_layer_model(8, 2, 2, 4, 8, 8)
    for w in (O.L_WO, O.L_WD):
        r, k = m.shape(O.layer_tid(0, w))
        m.set_tensor(O.layer_tid(0, w), np.zeros(r * k))
    m.set_tensor(O.T_LMHEAD, np.eye(8))
    toks = np.array([1, 5, 2], dtype=np.int32)
    out = O.forward(m, O.Cache(m, 8, 8), toks, np.arange(3), want_logits=True)
    x = m.get_tensor(O.T_EMBED).reshape(8, 8)[toks]
    h = np.stack([r * (1.0 / math.sqrt(float(np.dot(r, r)) / 8 + cfg.rms_eps)) for r in x])
    assert np.max(np.abs(h - _bf(h))) > 1e-4              # the rounding is visible in this case
    assert np.allclose(out.logits, _bf(h), rtol=0, atol=1e-12)


def test_bf16_rounding_points_of_the_attention_block():
    """bf16 model, d = hd = 2, one head, two tokens; W_q = I, W_k = [[0.75, 0], [0, 0]], W_v = 0.75 I,
    W_o = I, MLP zero. Token 1 = (0, 1) has key 0 exactly, so row 1's softmax over keys {0, 1} has
    the closed form p0 = e^s / (e^s + 1), s = q1 . k0 / sqrt(2). q, k and v are rounded to bf16
    after the rotary embedding, and so is the attention output."""
    cfg, m = _bf16_layer_model(2, 1, 1, 2, 2, 4)
    A, B = np.array([1.0625, 0.3125]), np.array([0.0, 1.0])
    E = np.zeros((4, 2))
    E[0], E[1], E[2], E[3] = A, B, [0.5, 0.25], [-1.0, 2.0]
    m.set_tensor(O.T_EMBED, E.ravel())
    m.set_tensor(O.layer_tid(0, O.L_WQ), np.eye(2).ravel())
    m.set_tensor(O.layer_tid(0, O.L_WK), np.array([0.75, 0.0, 0.0, 0.0]))
    m.set_tensor(O.layer_tid(0, O.L_WV), (0.75 * np.eye(2)).ravel())
    m.set_tensor(O.layer_tid(0, O.L_WO), np.eye(2).ravel())
    for w in (O.L_WG, O.L_WU, O.L_WD):
        m.set_tensor(O.layer_tid(0, w), np.zeros(4))
    out = O.forward(m, O.Cache(m, 8, 8), np.array([0, 1], dtype=np.int32), np.arange(2), want_hidden=True)

    def norm(x):
        return _bf(x * (1.0 / math.sqrt(float(np.dot(x, x)) / 2 + cfg.rms_eps)))

    h0, h1 = norm(A), norm(B)
    c, sn = math.cos(1.0), math.sin(1.0)                      # position 1, frequency theta^0 = 1
    q1 = _bf(np.array([h1[0] * c - h1[1] * sn, h1[1] * c + h1[0] * sn]))
    k0 = _bf(np.array([0.75 * h0[0], 0.0]))                   # position 0: no rotation
    assert abs(k0[0] - 0.75 * h0[0]) > 1e-4                    # the key needs rounding in this case
    v0, v1 = _bf(0.75 * h0), _bf(0.75 * h1)
    s = (q1[0] * k0[0] + q1[1] * k0[1]) * (1.0 / math.sqrt(2.0))
    mx = max(s, 0.0)
    p0, p1 = math.exp(s - mx), math.exp(0.0 - mx)
    att1 = _bf((p0 * v0 + p1 * v1) / (p0 + p1))
    assert np.max(np.abs(att1 - (p0 * v0 + p1 * v1) / (p0 + p1))) > 1e-4
    assert np.allclose(out.hidden[0], A + v0, rtol=0, atol=1e-12)   # row 0 sees only itself
    assert np.allclose(out.hidden[1], B + att1, rtol=0, atol=1e-12)


def test_bf16_swiglu_product_is_rounded():
    """bf16 model, attention output zero, W_gate = I, W_up = 2 I, W_down = 3 I: the hidden state is
    x + 3 bf16(silu(h) 2h) with h the bf16 RMSNorm output."""
    cfg, m = _bf16_layer_model(6, 2, 2, 2, 6, 16)
    r, k = m.shape(O.layer_tid(0, O.L_WO))
    m.set_tensor(O.layer_tid(0, O.L_WO), np.zeros(r * k))
    for w, sc in ((O.L_WG, 1.0), (O.L_WU, 2.0), (O.L_WD, 3.0)):
        m.set_tensor(O.layer_tid(0, w), sc * np.eye(6))
    toks = np.array([1, 9, 4], dtype=np.int32)
    out = O.forward(m, O.Cache(m, 8, 8), toks, np.arange(3), want_hidden=True)
    x = m.get_tensor(O.T_EMBED).reshape(16, 6)[toks]
    h = _bf(np.stack([r * (1.0 / math.sqrt(float(np.dot(r, r)) / 6 + cfg.rms_eps)) for r in x]))
    silu = np.vectorize(lambda t: t / (1.0 + math.exp(-t)))
    prod = silu(h) * (2.0 * h)
    assert np.max(np.abs(prod - _bf(prod))) > 1e-4
    assert np.allclose(out.hidden, x + 3.0 * _bf(prod), rtol=0, atol=1e-12)


def test_bf16_kv_cache_holds_bf16_values():
    """The KV cache of a bf16 model is bf16 (the precision the kernels store pages in): every committed
    K (after the rotary embedding) and V value equals its own bf16 rounding, while the same entries of
    the fp32 model do not all do so."""
    for bf16 in (True, False):
        cfg = O.ModelConfig(n_layers=2, d_model=64, n_heads=4, n_kv_heads=2, head_dim=16, d_ff=96, vocab=64,
                            bf16=bf16)
        m = O.Model(cfg).init_random(9, 0.3)
        c = O.Cache(m, 16, 16)
        toks = I.prompt_tokens(cfg.vocab, 7, seed=5)
        O.forward(m, c, toks, np.arange(7))
        c.commit(np.arange(7, dtype=np.int32))
        vals = np.concatenate([c.entry(l, w, p).ravel() for l in range(2) for w in (0, 1) for p in range(7)])
        assert np.count_nonzero(vals) > 0.9 * vals.size
        if bf16:
            assert np.array_equal(vals, _bf(vals))
        else:
            assert not np.array_equal(vals, _bf(vals))


# ------------------------------------------------------------------------------------------
# Rounding-noise diagnostic (sizes the logit tolerance of wide bf16 models)
# ------------------------------------------------------------------------------------------
def test_perturbation_is_off_by_default_and_switches_back_off():
    m16 = _tiny(bf16=True)
    toks = I.prompt_tokens(4096, 8, seed=12)

    def run():
        return O.forward(m16, O.Cache(m16, 16, 8), toks, np.arange(8), want_logits=True).logits

    a = run()
    O.set_perturbation(2.0 ** -12, 3)
    b = run()
    O.set_perturbation(0.0)
    c = run()
    assert np.array_equal(a, c)
    assert not np.array_equal(a, b)          # the hook is applied (a few roundings flip) ...
    assert np.abs(a - b).max() < 5e-2        # ... and moves a tiny model's logits by little


def test_perturbation_acts_at_the_bf16_rounding_points_only():
    """An fp32 model has no bf16 rounding point, so the diagnostic leaves it unchanged; a bf16 model
    perturbed by a relative 2^-7 (half a bf16 unit at most) moves, by rounding flips, far more than
    the same model at 2^-24."""
    m32 = _tiny(bf16=False)
    m16 = _tiny(bf16=True)
    toks = I.prompt_tokens(4096, 8, seed=13)

    def run(m):
        return O.forward(m, O.Cache(m, 16, 8), toks, np.arange(8), want_logits=True).logits

    a32 = run(m32)
    a16 = run(m16)
    O.set_perturbation(2.0 ** -7, 4)
    b32 = run(m32)
    big = np.abs(run(m16) - a16).max()
    O.set_perturbation(2.0 ** -24, 4)
    small = np.abs(run(m16) - a16).max()
    O.set_perturbation(0.0)
    assert np.array_equal(a32, b32)
    assert big > 10 * small
