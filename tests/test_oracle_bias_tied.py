"""Pins of the oracle's Q/K/V biases and tied embeddings (the Qwen2.5 architecture's options), no GPU.

* tensor layout: biases exist only with qkv_bias (ids 9-11 of a layer: [1, Hq hd], [1, Hkv hd]
  twice), the LM head only without tie_embeddings;
* zero biases leave every output of the same weights exactly as without biases;
* b_v enters the values, unrotated: with Wv = 0 every row attends to the constant b_v, so the
  attention output is b_v for both query heads (GQA) — a closed form;
* b_q and b_k enter before the rotary embedding: with Wq = Wk = 0 and b_q = b_k = a e_0 the score
  of row p against key j is a^2 cos(p - j) / sqrt(hd) (the first rotary pair turns at rate 1);
  added after the rotation the scores would be constant, and a missing bias makes them zero;
* a tied model equals the untied one whose LM head is a copy of the embedding.
"""
import numpy as np
import pytest

from oracle import oracle as O

TINY = dict(n_layers=1, d_model=8, n_heads=2, n_kv_heads=1, head_dim=4, d_ff=4, vocab=32)


def _one_layer(seed, **kw):
    cfg = O.ModelConfig(**TINY, **kw)
    m = O.Model(cfg).init_random(seed, 0.5)
    m.set_tensor(O.layer_tid(0, O.L_WO), np.eye(8))
    m.set_tensor(O.layer_tid(0, O.L_WD), np.zeros(8 * 4))  # no MLP contribution
    return cfg, m


def test_tensor_layout():
    plain = O.Model(O.ModelConfig(**TINY))
    bt = O.Model(O.ModelConfig(**TINY, qkv_bias=True, tie_embeddings=True))
    for w in (O.L_BQ, O.L_BK, O.L_BV):
        with pytest.raises(ValueError):
            plain.shape(O.layer_tid(0, w))
    assert bt.shape(O.layer_tid(0, O.L_BQ)) == (1, 8)
    assert bt.shape(O.layer_tid(0, O.L_BK)) == (1, 4)
    assert bt.shape(O.layer_tid(0, O.L_BV)) == (1, 4)
    assert plain.shape(O.T_LMHEAD) == (32, 8)
    with pytest.raises(ValueError):
        bt.shape(O.T_LMHEAD)
    # random biases are drawn like the matrices (nonzero, of the requested scale)
    bt.init_random(5, 0.5)
    b = bt.get_tensor(O.layer_tid(0, O.L_BQ))
    assert np.all(b != 0) and 0.05 < np.std(b) < 2.0


def test_zero_biases_change_nothing():
    for bf16 in (False, True):
        cfg = dict(TINY, n_layers=2, vocab=64, bf16=bf16)
        a = O.Model(O.ModelConfig(**cfg)).init_random(11, 0.3)
        b = O.Model(O.ModelConfig(**cfg, qkv_bias=True)).init_random(11, 0.3)
        for l in range(2):
            for w in (O.L_BQ, O.L_BK, O.L_BV):
                r, k = b.shape(O.layer_tid(l, w))
                b.set_tensor(O.layer_tid(l, w), np.zeros(r * k))
        toks = np.array([5, 1, 60, 7, 7, 33], dtype=np.int32)
        ra = O.forward(a, O.Cache(a, 16, 8), toks, np.arange(6), want_logits=True, want_hidden=True)
        rb = O.forward(b, O.Cache(b, 16, 8), toks, np.arange(6), want_logits=True, want_hidden=True)
        assert np.array_equal(ra.logits, rb.logits) and np.array_equal(ra.hidden, rb.hidden)


def test_value_bias_closed_form():
    cfg, m = _one_layer(3, qkv_bias=True)
    c = np.array([0.5, -1.25, 2.0, 0.75])
    m.set_tensor(O.layer_tid(0, O.L_WV), np.zeros(4 * 8))
    m.set_tensor(O.layer_tid(0, O.L_BV), c)
    toks = np.array([3, 17, 5, 5, 30], dtype=np.int32)
    out = O.forward(m, O.Cache(m, 8, 8), toks, np.arange(5), want_hidden=True)
    x = m.get_tensor(O.T_EMBED).reshape(32, 8)[toks]
    assert np.allclose(out.hidden, x + np.concatenate([c, c])[None, :], rtol=0, atol=1e-13)


def test_query_key_biases_enter_before_the_rotation():
    cfg, m = _one_layer(4, qkv_bias=True)
    a = 1.75  # exact in fp32, the storage precision of this model
    m.set_tensor(O.layer_tid(0, O.L_WQ), np.zeros(8 * 8))
    m.set_tensor(O.layer_tid(0, O.L_WK), np.zeros(4 * 8))
    m.set_tensor(O.layer_tid(0, O.L_BQ), np.array([a, 0, 0, 0, a, 0, 0, 0]))
    m.set_tensor(O.layer_tid(0, O.L_BK), np.array([a, 0, 0, 0]))
    m.set_tensor(O.layer_tid(0, O.L_WV), np.hstack([np.eye(4), np.zeros((4, 4))]))
    m.set_tensor(O.layer_tid(0, O.L_BV), np.zeros(4))
    toks = np.array([3, 17, 5, 9, 30, 2], dtype=np.int32)
    pos = np.arange(6)
    out = O.forward(m, O.Cache(m, 8, 8), toks, pos, want_hidden=True)
    x = m.get_tensor(O.T_EMBED).reshape(32, 8)[toks]
    h = x / np.sqrt(np.mean(x * x, axis=1, keepdims=True) + cfg.rms_eps)
    for i in range(6):
        s = a * a * np.cos(pos[i] - pos[: i + 1]) / 2.0   # 1 / sqrt(hd) = 1/2
        w = np.exp(s - s.max())
        w /= w.sum()
        att = w @ h[: i + 1, :4]
        assert np.allclose(out.hidden[i], x[i] + np.concatenate([att, att]), rtol=0, atol=1e-12)


def test_tied_equals_untied_with_the_embedding_as_head():
    for bf16 in (False, True):
        cfg = dict(TINY, n_layers=2, vocab=64, bf16=bf16)
        t = O.Model(O.ModelConfig(**cfg, tie_embeddings=True)).init_random(12, 0.3)
        u = O.Model(O.ModelConfig(**cfg)).init_random(12, 0.3)
        u.set_tensor(O.T_LMHEAD, t.get_tensor(O.T_EMBED))
        toks = np.array([5, 1, 60, 7, 33], dtype=np.int32)
        rt = O.forward(t, O.Cache(t, 16, 8), toks, np.arange(5), want_logits=True)
        ru = O.forward(u, O.Cache(u, 16, 8), toks, np.arange(5), want_logits=True)
        assert np.array_equal(rt.logits, ru.logits) and np.array_equal(rt.argmax, ru.argmax)
