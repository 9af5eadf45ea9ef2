"""Pins of the oracle's grouped-query attention (the Dream-7B model the paper also runs, Sec. 5.1:
fewer K/V heads than query heads; query head h reads K/V head h / (H / Hkv)).

- GQA equals multi-head attention whose K/V projection repeats each K/V head's weights for the
  query heads of its group (bit-exact: same products, same order); a wrong head mapping (h % Hkv
  instead of h / G, say) fails it.
- One GQA layer against a float64 numpy restatement of the LLaDA layer (RMSNorm, rotate-half
  RoPE, bidirectional softmax attention with grouped K/V, SwiGLU, untied head).
- n_kv_heads = n_heads is the multi-head path, bit-exact.
- The session's prefix K/V cache holds the K/V heads only and equals the forward's K/V.
"""
import numpy as np
import pytest

import dllm_inputs as I
import oracle as O

TINY_GQA = dict(n_layers=2, d_model=256, n_heads=4, head_dim=64, ffn=688, vocab=1024, mask_id=1023,
                rope_base=10000.0)


@pytest.fixture(scope="module")
def lib(oracle_lib):
    return oracle_lib


def _f32(bits):
    return (bits.astype(np.uint32) << 16).view(np.float32)


def test_gqa_equals_mha_with_repeated_kv_weights(lib):
    gqa = O.Model(O.OracleConfig(**TINY_GQA, n_kv_heads=2))
    mha = O.Model(O.OracleConfig(**TINY_GQA), zero=True)
    H, hd, G = 4, 64, 2
    for which in (O.T_EMBED, O.T_HEAD):
        mha.weight(-1, which)[:] = gqa.weight(-1, which)
    for layer in range(2):
        for w in (O.W_Q, O.W_O, O.W_GATE, O.W_UP, O.W_DOWN):
            mha.weight(layer, w)[:] = gqa.weight(layer, w)
        for w in (O.W_K, O.W_V):
            src, dst = gqa.weight(layer, w), mha.weight(layer, w)
            assert src.shape == (2 * hd, 256) and dst.shape == (4 * hd, 256)
            for h in range(H):
                dst[h * hd:(h + 1) * hd] = src[(h // G) * hd:(h // G + 1) * hd]
    tok = I.uniform_prompt(24, 1024, 1023, seed=5)
    pos = np.arange(24, dtype=np.int32)
    a = O.forward(gqa, tok, pos, want_kv=True)
    b = O.forward(mha, tok, pos, want_kv=True)
    assert np.array_equal(a["logits"], b["logits"])
    for h in range(H):
        assert np.array_equal(b["k"][:, :, h * hd:(h + 1) * hd], a["k"][:, :, (h // G) * hd:(h // G + 1) * hd])
        assert np.array_equal(b["v"][:, :, h * hd:(h + 1) * hd], a["v"][:, :, (h // G) * hd:(h // G + 1) * hd])
    # the grouping matters: K/V heads differ, so pairing query head 1 with K/V head 1 changes logits
    for h in (1, 2):
        src = gqa.weight(0, O.W_K)
        mha.weight(0, O.W_K)[h * hd:(h + 1) * hd] = src[(h % 2) * hd:(h % 2 + 1) * hd]
    c = O.forward(mha, tok, pos)
    assert not np.array_equal(a["logits"], c["logits"])


def _np_forward(model, cfg, tok, pos):
    d, H, hd, Hkv = cfg["d_model"], cfg["n_heads"], cfg["head_dim"], cfg["n_kv_heads"]
    G = H // Hkv
    W = lambda l, w: _f32(model.weight(l, w)).astype(np.float64)  # noqa: E731
    x = _f32(model.weight(-1, O.T_EMBED))[tok].astype(np.float64)
    T = len(tok)
    th = cfg["rope_base"] ** (-2.0 * np.arange(hd // 2) / hd)
    ang = pos[:, None].astype(np.float64) * th[None, :]
    cs, sn = np.cos(ang)[:, None, :], np.sin(ang)[:, None, :]

    def norm(v):
        return v / np.sqrt((v * v).mean(1, keepdims=True) + 1e-5)

    def rope(v):
        a, b = v[..., :hd // 2], v[..., hd // 2:]
        return np.concatenate([a * cs - b * sn, b * cs + a * sn], -1)

    for layer in range(cfg["n_layers"]):
        h = norm(x)
        q = rope((h @ W(layer, O.W_Q).T).reshape(T, H, hd))
        k = rope((h @ W(layer, O.W_K).T).reshape(T, Hkv, hd))
        v = (h @ W(layer, O.W_V).T).reshape(T, Hkv, hd)
        att = np.empty((T, H, hd))
        for hh in range(H):
            s = q[:, hh] @ k[:, hh // G].T / np.sqrt(hd)
            p = np.exp(s - s.max(1, keepdims=True))
            att[:, hh] = (p / p.sum(1, keepdims=True)) @ v[:, hh // G]
        x = x + att.reshape(T, H * hd) @ W(layer, O.W_O).T
        h = norm(x)
        g, u = h @ W(layer, O.W_GATE).T, h @ W(layer, O.W_UP).T
        x = x + (g / (1 + np.exp(-g)) * u) @ W(layer, O.W_DOWN).T
    return norm(x) @ W(-1, O.T_HEAD).T


def test_gqa_layer_matches_numpy(lib):
    cfg = dict(TINY_GQA, n_layers=1, n_kv_heads=1)
    model = O.Model(O.OracleConfig(**cfg))
    tok = I.uniform_prompt(20, 1024, 1023, seed=9)
    pos = np.arange(7, 27, dtype=np.int32)
    got = O.forward(model, tok, pos)["logits"]
    ref = _np_forward(model, cfg, tok, pos)
    assert np.abs(got - ref).max() <= 1e-5 * np.abs(ref).max()


def test_gqa_with_all_heads_is_multi_head(lib):
    a = O.Model(O.OracleConfig(**TINY_GQA))
    b = O.Model(O.OracleConfig(**TINY_GQA, n_kv_heads=4))
    tok = I.uniform_prompt(16, 1024, 1023, seed=3)
    pos = np.arange(16, dtype=np.int32)
    assert np.array_equal(O.forward(a, tok, pos)["logits"], O.forward(b, tok, pos)["logits"])


def test_gqa_session_prefix_cache_holds_kv_heads(lib):
    cfg = O.OracleConfig(**TINY_GQA, n_kv_heads=2)
    model = O.Model(cfg)
    prompt = I.uniform_prompt(40, 1024, 1023, seed=4)
    sess = O.Session(model, O.OracleSched(steps_per_block=8), prompt, 32)
    sess.prefill()
    f = O.forward(model, prompt, np.arange(40, dtype=np.int32), want_kv=True, logits=False)
    for layer in range(2):
        assert sess.prefix_kv(layer, 0).shape == (40, 128)
        assert np.array_equal(sess.prefix_kv(layer, 0), f["k"][layer])
        assert np.array_equal(sess.prefix_kv(layer, 1), f["v"][layer])
    sess.begin_block()
    for _ in range(8):
        out = sess.step()
    assert out["block_done"] == 1 and sess.begin_block() is False
    assert sess.state()[2] == 72
