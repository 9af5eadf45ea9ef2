"""Oracle parity of the configuration the benchmark times, at full depth, on the GPU.

LLaDA-8B shape (32 layers, d 4096, 32 heads x 128, ffn 12288, vocab 126464),
batch 1: a 512-token uniform prompt prefilled into the prefix KV cache, then one
denoising step on a 32-token window with 24 positions masked (Sec. 2.1,
block-wise decoding with the prefix KV cache), in the context configuration and
launch path `bench.py` uses.  The oracle runs the same prefill and the same step
from the same (teacher-forced) window state.

Tolerances.  A randomly initialised 32-layer model amplifies any bf16-sized
difference in its hidden state layer after layer, so no computation with bf16
operands stays within 1e-2 of the fp32 oracle at depth.  Each bound below is
therefore max(1e-2, 2 u A): u = 2^-8 (bf16's unit roundoff) and A the oracle's
own amplification of a perturbation of its input at that layer or logit row,
from tests/golden/llada8b_depth_sensitivity.json (written by the oracle alone).
Checked:
  - the prefix K/V that the 512-token prefill leaves in the cache, at the first,
    a middle and the last layer;
  - the step's logits over the whole vocabulary, row by row;
  - the fused LM head's argmax equal to the argmax of the GPU's own logits, and
    to the oracle's wherever the oracle's top-1/top-2 margin exceeds twice the
    row's largest logit deviation (no smaller deviation can flip it);
  - the commit: one position, the mask never committed; where the oracle's most
    confident masked position leads the runner-up by more than the logit
    deviation allows, the GPU's new state equals the oracle's exactly, otherwise
    the GPU's pick is one of the near-tied positions, carries the GPU's argmax,
    and nothing else changed.
The oracle needs a few minutes on the host cores (about 7 TFLOP for the
prefill at fp64 accumulation).
"""
import json
import os

import numpy as np
import pytest

import dllm_inputs as I
import oracle as O

torch = pytest.importorskip("torch")
pytestmark = [pytest.mark.gpu, pytest.mark.slow]

SHAPE = dict(n_layers=32, d_model=4096, n_heads=32, head_dim=128, ffn=12288, vocab=126464, mask_id=126463,
             rope_base=500000.0)
LP, T, MASKED = 512, 32, 24
U_BF16 = 2.0 ** -8
GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden", "llada8b_depth_sensitivity.json")


def _tol(amplification):
    return max(1e-2, 2.0 * U_BF16 * amplification)


def _window_state(tok, st, mask_id, committed, masked):
    win = np.arange(LP, LP + T)
    tok = tok.copy()
    st = st.copy()
    tok[win] = I.uniform_prompt(T, SHAPE["vocab"], mask_id, seed=7)
    st[win] = committed
    m = win[I.masked_positions(T, MASKED)]
    tok[m], st[m] = mask_id, masked
    return tok, st


def test_llada8b_bench_configuration_full_depth_matches_oracle():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    import paper_2606_13740_gb300 as pkg
    pkg.lib()
    prompt = I.uniform_prompt(LP, SHAPE["vocab"], SHAPE["mask_id"], seed=I.SEED_PROMPT)

    # GPU: the benchmark's context and schedule
    ctx = pkg.Context(pkg.Config(max_batch=1, max_ctx=LP + T, max_window=LP, **SHAPE))
    ctx.dllm_prefill(pkg.Sched(steps_per_block=MASKED), prompt, T)
    ctx.dllm_begin_block()
    g_tok, g_st, _ = ctx.dllm_get_state()
    w_tok, w_st = _window_state(g_tok[0], g_st[0], SHAPE["mask_id"], pkg.COMMITTED, pkg.MASKED)
    ctx.dllm_set_state(w_tok[None], w_st[None])
    ctx.dllm_set_debug(1)  # materialise the logits
    gout = ctx.dllm_denoise_step()
    gd = ctx.dllm_get_step_debug(logits=True)
    g_after = ctx.dllm_get_state()
    g_kv = {(l, w): ctx.dllm_get_kv(l, w, 0, 0, LP) for l in (0, 15, 31) for w in (0, 1)}
    ctx.close()

    # oracle: the same prefill and step
    model = O.Model(O.OracleConfig(**SHAPE))
    sess = O.Session(model, O.OracleSched(steps_per_block=MASKED), prompt, T)
    sess.prefill()
    assert sess.begin_block()
    o_tok, o_st, _ = sess.state()
    assert np.array_equal(o_tok, g_tok[0]) and np.array_equal(o_st, g_st[0])
    sess.set_state(w_tok, w_st)
    oout = sess.step(keep_logits=True)
    od = sess.decisions(logits=True)
    o_after_tok, o_after_st, o_kv_len = sess.state()
    assert o_kv_len == LP
    with open(GOLDEN) as f:
        sens = json.load(f)
    for (l, w), got in g_kv.items():
        ref = sess.prefix_kv(l, w)
        rel = np.linalg.norm(got - ref) / np.linalg.norm(ref)
        assert rel <= _tol(sens["A_K" if w == 0 else "A_V"][l]), (l, w, rel)
    del model, sess

    # logits, row by row
    lg, lo = gd["logits"][0], od["logits"]
    rel_rows = np.linalg.norm(lg - lo, axis=1) / np.linalg.norm(lo, axis=1)
    for r in range(T):
        assert rel_rows[r] <= _tol(sens["A_logits_rows"][r]), (r, rel_rows[r])
    # the fused head's argmax against the GPU's own logits, and against the oracle's where the
    # deviation cannot flip it
    own = lg.copy()
    own[:, SHAPE["mask_id"]] = -np.inf
    assert np.array_equal(gd["x0"][0], own.argmax(1))
    dev = np.abs(lg - lo).max(axis=1)
    safe = od["margin"] > 2 * dev
    assert np.array_equal(gd["x0"][0][safe], od["x0"][safe])
    assert not (gd["x0"][0] == SHAPE["mask_id"]).any()

    # the commit (one position: ceil(24 / 24))
    assert gout["n_committed"] == oout["n_committed"] == 1
    assert gout["masked_after"] == oout["masked_after"] == MASKED - 1
    masked_w = np.flatnonzero(w_st[LP:LP + T] == pkg.MASKED)
    conf = od["conf"][masked_w]
    order = np.argsort(-conf, kind="stable")
    lead = (conf[order[0]] - conf[order[1]]) / conf[order[0]]
    # a logit deviation of at most e moves a confidence by at most a factor exp(2e)
    tol = np.expm1(4 * float(dev[masked_w].max()))
    g_new = np.flatnonzero((g_after[1][0] != w_st) & (w_st == pkg.MASKED))
    o_new = np.flatnonzero((o_after_st != w_st) & (w_st == pkg.MASKED))
    assert len(g_new) == len(o_new) == 1
    p = g_new[0]
    assert g_after[1][0][p] == pkg.COMMITTED and g_after[0][0][p] == gd["x0"][0][p - LP]
    if lead > tol:
        assert np.array_equal(g_after[0][0], o_after_tok) and np.array_equal(g_after[1][0], o_after_st)
    else:
        assert od["conf"][p - LP] >= conf[order[0]] * (1 - tol) / (1 + tol)
        unchanged = np.ones(LP + T, bool)
        unchanged[[p, o_new[0]]] = False
        assert np.array_equal(g_after[0][0][unchanged], o_after_tok[unchanged])
        assert np.array_equal(g_after[1][0][unchanged], o_after_st[unchanged])
