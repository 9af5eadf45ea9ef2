"""Grouped-query attention on the GPU (the Dream-7B model the paper also runs, Sec. 5.1: fewer
K/V heads than query heads), through the C ABI, against the oracle.

- Seeded weights bit-exact with the oracle's (the fused QKV matrix holds qd + 2 kvd rows).
- The attention kernels (mma.sync below 1024 keys, tcgen05 above) against float64 numpy with
  query head h reading K/V head h / (H / Hkv).
- A tiny GQA model's block loop teacher-forced on the oracle (logits relative L2 <= 1e-2,
  argmax where the margin exceeds 0.05, bookkeeping bit-exact), then its prefix K/V cache.
- A Dream-7B-shaped model (d 3584, 28 query heads, 4 K/V heads of 128, ffn 18944, vocab
  152064) with two layers: prefill and two teacher-forced steps against the oracle.
"""
import numpy as np
import pytest

import dllm_inputs as I
import oracle as O

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

TINY_GQA = dict(n_layers=2, d_model=256, n_heads=4, head_dim=64, ffn=688, vocab=1024, mask_id=1023,
                rope_base=10000.0, n_kv_heads=2)
DREAM = dict(d_model=3584, n_heads=28, head_dim=128, ffn=18944, vocab=152064, mask_id=152063, rope_base=1000000.0,
             n_kv_heads=4)


@pytest.fixture(scope="module")
def pkg():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    import paper_2606_13740_gb300 as p
    p.lib()
    return p


def _f64(t):
    return t.float().cpu().numpy().astype(np.float64)


@pytest.mark.parametrize("B,T,H,Hkv,hd,kv,cap", [
    (1, 32, 4, 2, 64, [300], 400), (2, 40, 8, 1, 128, [5, 700], 800),      # mma.sync kernel
    (2, 64, 8, 2, 128, [1100, 1500], 1600), (1, 32, 28, 4, 128, [2000], 2048),  # tcgen05 kernel
])
def test_gqa_attention_matches_numpy(pkg, B, T, H, Hkv, hd, kv, cap):
    dev = torch.device("cuda:0")
    rng = np.random.default_rng(B * 7 + H + Hkv)
    bf = lambda s: torch.from_numpy(rng.standard_normal(s).astype(np.float32)).to(torch.bfloat16)  # noqa: E731
    q, k, v = bf((B, H, T, hd)), bf((B, Hkv, cap, hd)), bf((B, Hkv, cap, hd))
    kv_len = torch.tensor(kv, dtype=torch.int32)
    out = pkg.dllm_op_attention(q.to(dev), k.to(dev), v.to(dev), kv_len.to(dev), B, T, H, hd, cap, max(kv),
                                Hkv=Hkv)
    got = out.float().cpu().numpy()
    qf, kf, vf = _f64(q), _f64(k), _f64(v)
    ref = np.zeros((B * T, H * hd))
    for b in range(B):
        nk = kv[b] + T
        for h in range(H):
            s = qf[b, h] @ kf[b, h // (H // Hkv), :nk].T / np.sqrt(hd)
            p = np.exp(s - s.max(1, keepdims=True))
            ref[b * T:(b + 1) * T, h * hd:(h + 1) * hd] = (p / p.sum(1, keepdims=True)) @ vf[b, h // (H // Hkv), :nk]
    rel = np.linalg.norm(got - ref) / np.linalg.norm(ref)
    assert rel <= 1e-2, rel


def test_gqa_weights_bit_exact(pkg):
    model = O.Model(O.OracleConfig(**TINY_GQA))
    ctx = pkg.Context(pkg.Config(max_ctx=128, max_window=64, **TINY_GQA))
    for layer in range(2):
        for w in range(7):
            assert np.array_equal(ctx.dllm_get_weight(layer, w), model.weight(layer, w)), (layer, w)
    ctx.close()


def test_gqa_blockwise_teacher_forced(pkg):
    from test_gpu_step import _run_teacher_forced
    model = O.Model(O.OracleConfig(**TINY_GQA))
    prompt = I.uniform_prompt(64, 1024, 1023, seed=21)
    ctx = pkg.Context(pkg.Config(max_ctx=256, max_window=160, **TINY_GQA))
    kw = dict(steps_per_block=8, theta_remask=0.5, remask_max=1, spec_blocks=1, spec_trigger=16)
    sess, steps, worst = _run_teacher_forced(model, O.OracleSched(**kw), pkg.Sched(**kw), prompt, 96, ctx)
    assert steps >= 24
    kv_len = sess.state()[2]
    for layer in range(2):
        for which in (0, 1):
            ref = sess.prefix_kv(layer, which)
            got = ctx.dllm_get_kv(layer, which, 0, 0, kv_len)
            assert got.shape == ref.shape == (kv_len, 128)
            assert np.linalg.norm(got - ref) / np.linalg.norm(ref) <= 1e-2
    ctx.close()


def test_dream7b_shape_two_layers_teacher_forced(pkg):
    ocfg = O.OracleConfig(n_layers=2, **DREAM)
    model = O.Model(ocfg)
    ctx = pkg.Context(pkg.Config(n_layers=2, max_ctx=128, max_window=64, **DREAM))
    for w in (0, 1, 2):
        assert np.array_equal(ctx.dllm_get_weight(1, w), model.weight(1, w)), w
    prompt = I.uniform_prompt(64, ocfg.vocab, ocfg.mask_id)
    sess = O.Session(model, O.OracleSched(steps_per_block=32), prompt, 32)
    sess.prefill()
    sess.begin_block()
    ctx.dllm_prefill(pkg.Sched(steps_per_block=32), prompt, 32)
    ctx.dllm_set_debug(1)
    ctx.dllm_begin_block()
    for _ in range(2):
        oo = sess.step(keep_logits=True)
        go = ctx.dllm_denoise_step()
        od = sess.decisions(logits=True)
        gd = ctx.dllm_get_step_debug(logits=True)
        rel = np.linalg.norm(gd["logits"][0] - od["logits"]) / np.linalg.norm(od["logits"])
        assert rel <= 1e-2, rel
        safe = od["margin"] > 0.05
        assert safe.sum() > 0
        assert np.array_equal(gd["x0"][0][safe], od["x0"][safe])
        assert go["n_committed"] == oo["n_committed"] == 1
        tok, st, _ = sess.state()
        ctx.dllm_set_state(tok[None], st[None])
    for layer in (0, 1):
        for which in (0, 1):
            ref = sess.prefix_kv(layer, which)
            got = ctx.dllm_get_kv(layer, which, 0, 0, 64)
            assert got.shape == (64, 512)
            assert np.linalg.norm(got - ref) / np.linalg.norm(ref) <= 1e-2
    ctx.close()
