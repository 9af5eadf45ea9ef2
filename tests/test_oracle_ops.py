"""Pins of the oracle's transformer step (the LLaDA forward of Sec. 2.1 and
Sec. 5.1 "Models") against closed forms, invariants and library routines.

Each test builds special-case weights so that one part of the forward reduces
to something numpy/scipy computes independently (matmul, softmax, expit,
complex rotation), or checks an invariant the architecture guarantees
(unit RMS, RoPE relative-position invariance, no causal mask).
"""
import numpy as np
import pytest
from scipy.special import expit, softmax

import oracle as O

SMALL = O.OracleConfig(n_layers=1, d_model=16, n_heads=2, head_dim=8, ffn=24, vocab=32, mask_id=31,
                       rope_base=10000.0, rms_eps=1e-5, weight_seed=99)


def _bf16(x):
    return O.f32_to_bf16_bits(np.asarray(x, np.float32)).reshape(np.shape(x))


def _f(bits):
    return O.bf16_to_f32(bits).astype(np.float64)


def _rms(x, eps=1e-5):
    x = np.asarray(x, np.float64)
    return x / np.sqrt((x * x).mean(-1, keepdims=True) + eps)


def _zero_model(rng):
    m = O.Model(SMALL, zero=True)
    m.weight(-1, O.T_EMBED)[:] = _bf16(rng.standard_normal((SMALL.vocab, SMALL.d_model)) * 0.5)
    m.weight(-1, O.T_HEAD)[:] = _bf16(rng.standard_normal((SMALL.vocab, SMALL.d_model)) * 0.5)
    return m


def _eye(rows, cols):
    return _bf16(np.eye(rows, cols, dtype=np.float32))


def _head_logits(m, x):
    return _rms(x) @ _f(m.weight(-1, O.T_HEAD)).T


# ---------------------------------------------------------------- ops
def test_rmsnorm_unit_rms_and_scale_invariance(oracle_lib):
    rng = np.random.default_rng(1)
    x = rng.standard_normal(64).astype(np.float32) * 3
    g = np.ones(64, np.float32)
    y = O.rmsnorm(x, g, 0.0)
    assert abs(np.sqrt((y.astype(np.float64) ** 2).mean()) - 1.0) < 1e-6
    assert np.allclose(O.rmsnorm(x * 8, g, 0.0), y, rtol=1e-6)
    g2 = rng.random(64).astype(np.float32)
    assert np.allclose(O.rmsnorm(x, g2, 0.0), y * g2, rtol=1e-6)


def test_rope_is_complex_rotation(oracle_lib):
    rng = np.random.default_rng(2)
    hd, base = 16, 10000.0
    v = rng.standard_normal(hd).astype(np.float32)
    for pos in (0, 1, 7, 513):
        out = O.rope(v, base, pos)
        z = v[: hd // 2].astype(np.float64) + 1j * v[hd // 2:].astype(np.float64)
        theta = base ** (-np.arange(hd // 2) * 2.0 / hd)
        zr = z * np.exp(1j * pos * theta)
        want = np.concatenate([zr.real, zr.imag])
        assert np.allclose(out, want, rtol=1e-5, atol=1e-6)
    assert np.array_equal(O.rope(v, base, 0), v)


def test_rope_relative_position(oracle_lib):
    rng = np.random.default_rng(3)
    q = rng.standard_normal(32).astype(np.float32)
    k = rng.standard_normal(32).astype(np.float32)
    d1 = float(O.rope(q, 10000.0, 40) @ O.rope(k, 10000.0, 33))
    d2 = float(O.rope(q, 10000.0, 107) @ O.rope(k, 10000.0, 100))
    assert abs(d1 - d2) < 1e-4 * max(1.0, abs(d1))


def test_decide_against_scipy_softmax(oracle_lib):
    rng = np.random.default_rng(4)
    V, mask = 50, 49
    z = rng.standard_normal(V).astype(np.float32) * 2
    z[mask] = 100.0  # the mask id's own logit is the largest: still excluded
    x0, conf, tokconf, margin = O.decide(z, mask, cur=7)
    zz = z.astype(np.float64).copy()
    zz[mask] = -np.inf
    p = softmax(zz)
    assert x0 == int(np.argmax(zz)) and x0 != mask
    assert abs(conf - p[x0]) < 1e-6
    assert abs(tokconf - p[7]) < 1e-7
    assert abs(p.sum() - 1.0) < 1e-12
    srt = np.sort(zz[np.isfinite(zz)])
    assert abs(margin - (srt[-1] - srt[-2])) < 1e-6
    _, _, tc_mask, _ = O.decide(z, mask, cur=mask)
    assert tc_mask == 0.0


def test_decide_ties_and_uniform(oracle_lib):
    V, mask = 40, 0
    z = np.zeros(V, np.float32)
    x0, conf, _, margin = O.decide(z, mask, cur=3)
    assert x0 == 1  # lowest id that is not the mask
    assert abs(conf - 1.0 / (V - 1)) < 1e-7
    assert margin == 0.0
    z[5] = z[9] = 1.0
    assert O.decide(z, mask, cur=3)[0] == 5


# ---------------------------------------------------------------- forward
def test_forward_identity_layers_reduce_to_head(oracle_lib):
    """All projections zero: the residual stream is the embedding."""
    rng = np.random.default_rng(5)
    m = _zero_model(rng)
    tok = np.array([3, 17, 0, 25, 9], np.int32)
    out = O.forward(m, tok, np.arange(5))
    x = _f(m.weight(-1, O.T_EMBED))[tok]
    assert np.allclose(out["logits"], _head_logits(m, x), rtol=1e-5, atol=1e-5)


def test_forward_uniform_attention_is_mean_of_values(oracle_lib):
    """W_q = 0 gives equal scores: attention returns the mean value row over
    the cached prefix and the window (no causal mask)."""
    rng = np.random.default_rng(6)
    m = _zero_model(rng)
    d = SMALL.d_model
    wv = _bf16(rng.standard_normal((d, d)) * 0.3)
    m.weight(0, O.W_V)[:] = wv
    m.weight(0, O.W_O)[:] = _eye(d, d)
    tok = np.array([1, 2, 3, 4], np.int32)
    P = 3
    pk = rng.standard_normal((1, P, d)).astype(np.float32)
    pv = rng.standard_normal((1, P, d)).astype(np.float32)
    out = O.forward(m, tok, np.arange(P, P + 4), prefix_k=pk, prefix_v=pv, want_kv=True)
    x = _f(m.weight(-1, O.T_EMBED))[tok]
    v = _rms(x) @ _f(wv).T
    mean_v = np.concatenate([pv[0].astype(np.float64), v]).mean(0)
    assert np.allclose(out["v"][0], v, rtol=1e-5, atol=1e-6)
    assert np.allclose(out["logits"], _head_logits(m, x + mean_v), rtol=1e-4, atol=1e-5)


def test_forward_scores_match_scipy_softmax(oracle_lib):
    """Positions 0 (RoPE is the identity), W_q = W_k = W_v = W_o = I:
    per head, out_t = softmax(h_t . h_s / sqrt(hd)) h_s."""
    rng = np.random.default_rng(7)
    m = _zero_model(rng)
    d, H, hd = SMALL.d_model, SMALL.n_heads, SMALL.head_dim
    for w in (O.W_Q, O.W_K, O.W_V, O.W_O):
        m.weight(0, w)[:] = _eye(d, d)
    tok = np.array([4, 8, 15, 16, 23], np.int32)
    out = O.forward(m, tok, np.zeros(5, np.int32))
    x = _f(m.weight(-1, O.T_EMBED))[tok]
    h = _rms(x)
    att = np.zeros_like(h)
    for hh in range(H):
        sl = slice(hh * hd, (hh + 1) * hd)
        p = softmax(h[:, sl] @ h[:, sl].T / np.sqrt(hd), axis=1)
        att[:, sl] = p @ h[:, sl]
    assert np.allclose(out["logits"], _head_logits(m, x + att), rtol=1e-4, atol=1e-5)


def test_forward_swiglu(oracle_lib):
    """Attention off, W_g = W_u = I, W_d = I: x += silu(h) * h."""
    rng = np.random.default_rng(8)
    m = _zero_model(rng)
    d, F = SMALL.d_model, SMALL.ffn
    m.weight(0, O.W_GATE)[:] = _eye(F, d)
    m.weight(0, O.W_UP)[:] = _eye(F, d)
    m.weight(0, O.W_DOWN)[:] = _eye(d, F)
    tok = np.array([5, 6, 7], np.int32)
    out = O.forward(m, tok, np.arange(3))
    x = _f(m.weight(-1, O.T_EMBED))[tok]
    h = _rms(x)
    y = x + h * expit(h) * h
    assert np.allclose(out["logits"], _head_logits(m, y), rtol=1e-4, atol=1e-5)


def _random_model(layers=2):
    cfg = O.OracleConfig(n_layers=layers, d_model=64, n_heads=4, head_dim=16, ffn=96, vocab=128, mask_id=127,
                         weight_seed=1234)
    return O.Model(cfg)


def test_forward_rope_shift_invariance(oracle_lib):
    m = _random_model()
    tok = np.array([10, 20, 30, 40, 50, 60], np.int32)
    a = O.forward(m, tok, np.arange(6))["logits"]
    b = O.forward(m, tok, np.arange(6) + 300)["logits"]
    assert np.abs(a - b).max() < 1e-4 * np.abs(a).max()


def test_forward_permutation_equivariance_without_rope(oracle_lib):
    """Bidirectional attention: permuting the window permutes the outputs."""
    m = _random_model()
    tok = np.array([3, 14, 15, 92, 65, 35, 89], np.int32)
    perm = np.array([6, 2, 0, 5, 1, 4, 3])
    z = np.zeros(7, np.int32)
    a = O.forward(m, tok, z)["logits"]
    b = O.forward(m, tok[perm], z)["logits"]
    assert np.allclose(a[perm], b, rtol=1e-5, atol=1e-6)


def test_forward_no_causal_mask(oracle_lib):
    m = _random_model()
    tok = np.array([3, 14, 15, 92], np.int32)
    a = O.forward(m, tok, np.arange(4))["logits"]
    tok2 = tok.copy()
    tok2[-1] = 7
    b = O.forward(m, tok2, np.arange(4))["logits"]
    assert np.abs(a[0] - b[0]).max() > 1e-4  # the first position sees the last


def test_forward_group_mask_matches_separate_prefix(oracle_lib):
    """A two-group window (group 1 sees group 0, not vice versa) equals a
    forward over group 0 followed by group 1 attending to group 0's K/V."""
    m = _random_model()
    tok = np.array([5, 6, 7, 8, 9, 10, 11], np.int32)
    pos = np.arange(7)
    grp = np.array([0, 0, 0, 1, 1, 1, 1], np.int32)
    full = O.forward(m, tok, pos, group=grp, want_kv=True)
    first = O.forward(m, tok[:3], pos[:3], want_kv=True)
    second = O.forward(m, tok[3:], pos[3:], prefix_k=first["k"], prefix_v=first["v"], want_kv=True)
    assert np.array_equal(full["k"][:, :3], first["k"])
    assert np.array_equal(full["k"][:, 3:], second["k"])
    assert np.array_equal(full["logits"][3:], second["logits"])
