"""Parity at the LLaDA-8B shape on the GPU, through the C ABI.

- Full width, two layers (d 4096, 32 heads x 128, ffn 12288, vocab 126464):
  the oracle runs the same prefill and steps; logits within 1e-2 relative L2,
  argmax equal where the oracle's margin exceeds 0.05, teacher-forced.
- Full 32-layer model in the configuration the benchmark times (B=1, 512-token
  prompt, 32-token window with 24 masked): properties that hold at any size
  (exact commit count, mask never committed, bit-identical repeat after a
  rewind, prefix length unchanged) and seeded weights equal to the oracle's
  generator on sampled slices.
"""
import numpy as np
import pytest

import dllm_inputs as I
import oracle as O

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

SHAPE = dict(d_model=4096, n_heads=32, head_dim=128, ffn=12288, vocab=126464, mask_id=126463, rope_base=500000.0)


@pytest.fixture(scope="module")
def gpu():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    import paper_2606_13740_gb300 as pkg
    pkg.lib()
    return pkg


def test_full_width_two_layers_teacher_forced(gpu):
    ocfg = O.OracleConfig(n_layers=2, **SHAPE)
    model = O.Model(ocfg)
    ctx = gpu.Context(gpu.Config(n_layers=2, max_ctx=128, max_window=64, **SHAPE))
    for w in range(7):
        assert np.array_equal(ctx.dllm_get_weight(1, w), model.weight(1, w)), w
    prompt = I.uniform_prompt(64, ocfg.vocab, ocfg.mask_id)
    sess = O.Session(model, O.OracleSched(steps_per_block=32), prompt, 32)
    sess.prefill()
    sess.begin_block()
    ctx.dllm_prefill(gpu.Sched(steps_per_block=32), prompt, 32)
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


def test_llada8b_bench_configuration_properties(gpu):
    cfg = gpu.Config(n_layers=32, max_ctx=576, max_window=512, **SHAPE)
    ctx = gpu.Context(cfg)
    # seeded weights: sampled slices equal the oracle generator's definition
    wq = ctx.dllm_get_weight(31, 0)
    ref = O.gen_bf16(cfg.weight_seed, 16 + 8 * 31 + 0, 4096 * 1000, 4096 * 4, 0.02)
    assert np.array_equal(wq.reshape(-1)[4096 * 1000:4096 * 1004], ref)
    head = ctx.dllm_get_weight(-1, 2)
    ref = O.gen_bf16(cfg.weight_seed, O.T_HEAD, 4096 * 126000, 4096 * 8, 0.02)
    assert np.array_equal(head.reshape(-1)[4096 * 126000:4096 * 126008], ref)
    del head
    prompt = I.uniform_prompt(512, cfg.vocab, cfg.mask_id)
    sched = gpu.Sched(steps_per_block=24)
    ctx.dllm_prefill(sched, prompt, 32)
    ctx.dllm_begin_block()
    tok, st, _ = ctx.dllm_get_state()
    masked = I.masked_positions(32, 24)
    window = np.arange(512, 544)
    st[0, window] = gpu.COMMITTED
    tok[0, window] = I.uniform_prompt(32, cfg.vocab, cfg.mask_id, seed=7)
    st[0, window[masked]] = gpu.MASKED
    tok[0, window[masked]] = cfg.mask_id
    ctx.dllm_set_state(tok, st)  # also the rewind point
    out = ctx.dllm_denoise_step()
    assert out["n_committed"] == 1 and out["masked_after"] == 23  # ceil(24 / 24)
    d1 = ctx.dllm_get_step_debug()
    s1 = ctx.dllm_get_state()
    assert not (d1["x0"] == cfg.mask_id).any()
    assert s1[2][0] == 512
    newly = (s1[1][0] == gpu.COMMITTED) & (st[0] == gpu.MASKED)
    assert newly.sum() == 1 and s1[0][0][newly][0] == d1["x0"][0][np.flatnonzero(newly)[0] - 512]
    ctx.dllm_rewind_block()
    out2 = ctx.dllm_denoise_step()
    d2 = ctx.dllm_get_step_debug()
    assert out2 == out
    assert np.array_equal(d1["x0"], d2["x0"]) and np.array_equal(d1["conf"], d2["conf"])
    ctx.close()
