"""4-bit block-quantised weights on the GPU (the Q4_0 weights the paper runs, Sec. 5.1), through
the C ABI, against the oracle in the same format.

- The seeded 4-bit weights the device draws dequantise to exactly the oracle's bf16 values,
  for every projection and the LM head (tiny model; sampled rows at the LLaDA-8B width).
- The chained projections expand each 4-bit tile into bf16 on the fly: a tiny model's block
  loop teacher-forced on the oracle (logits relative L2 <= 1e-2, argmax where the margin
  exceeds 0.05, bookkeeping bit-exact) and its prefix K/V cache.
- Full LLaDA-8B width with two layers: prefill of 64 tokens and two teacher-forced steps.
"""
import numpy as np
import pytest

import dllm_inputs as I
import oracle as O

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

SHAPE_8B = dict(d_model=4096, n_heads=32, head_dim=128, ffn=12288, vocab=126464, mask_id=126463,
                rope_base=500000.0)


@pytest.fixture(scope="module")
def pkg():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    import paper_2606_13740_gb300 as p
    p.lib()
    return p


def test_q4_weights_dequantise_to_the_oracles(pkg):
    cfg = O.OracleConfig(weight_bits=4)
    model = O.Model(cfg)
    ctx = pkg.Context(pkg.Config(max_ctx=128, max_window=64, weight_bits=4))
    for layer in range(cfg.n_layers):
        for w in range(7):
            assert np.array_equal(ctx.dllm_get_weight(layer, w), model.weight(layer, w)), (layer, w)
    assert np.array_equal(ctx.dllm_get_weight(-1, 2), model.weight(-1, O.T_HEAD))
    assert np.array_equal(ctx.dllm_get_weight(-1, 1), model.weight(-1, O.T_EMBED))  # embedding stays bf16
    ctx.close()


@pytest.mark.parametrize("n_prompt", [64, 192])
def test_q4_blockwise_teacher_forced(pkg, n_prompt):
    """The 4-bit block loop against the oracle; a 192-token prompt puts the prefill on token
    tiles too wide for tensor-memory A stages (the shared-memory stages and their own rings)."""
    from test_gpu_step import _run_teacher_forced
    model = O.Model(O.OracleConfig(weight_bits=4))
    prompt = I.uniform_prompt(n_prompt, 1024, 1023, seed=31)
    ctx = pkg.Context(pkg.Config(max_ctx=n_prompt + 192, max_window=192, weight_bits=4))
    kw = dict(steps_per_block=8, theta_remask=0.5, remask_max=1, spec_blocks=1, spec_trigger=16)
    sess, steps, worst = _run_teacher_forced(model, O.OracleSched(**kw), pkg.Sched(**kw), prompt, 96, ctx)
    assert steps >= 24
    kv_len = sess.state()[2]
    for layer in range(2):
        for which in (0, 1):
            ref = sess.prefix_kv(layer, which)
            got = ctx.dllm_get_kv(layer, which, 0, 0, kv_len)
            assert np.linalg.norm(got - ref) / np.linalg.norm(ref) <= 1e-2
    ctx.close()


def test_q4_full_width_two_layers_teacher_forced(pkg):
    ocfg = O.OracleConfig(n_layers=2, weight_bits=4, **SHAPE_8B)
    model = O.Model(ocfg)
    ctx = pkg.Context(pkg.Config(n_layers=2, max_ctx=128, max_window=64, weight_bits=4, **SHAPE_8B))
    for w in (0, 4, 6):  # the fused QKV rows, the gate/up interleave, a K of 12288
        got, ref = ctx.dllm_get_weight(1, w), model.weight(1, w)
        rows = np.random.default_rng(w).choice(ref.shape[0], 64, replace=False)
        assert np.array_equal(got[rows], ref[rows]), w
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
        ref = sess.prefix_kv(layer, 0)
        got = ctx.dllm_get_kv(layer, 0, 0, 0, 64)
        assert np.linalg.norm(got - ref) / np.linalg.norm(ref) <= 1e-2
    ctx.close()
