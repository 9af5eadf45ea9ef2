"""End-to-end parity of the GPU denoising path with the oracle on the tiny
LLaDA-shaped config, through the C ABI: seeded weights bit-exact, and every
step teacher-forced on the oracle's state so the trajectories stay aligned.

Acceptance per step: logits relative L2 <= 1e-2 (bf16 path vs fp32 oracle);
argmax ids equal wherever the oracle's top-1/top-2 logit margin exceeds 0.05;
window, commit counts and token states bit-exact; committed positions equal
wherever the oracle's confidence ranking is unambiguous.
"""
import numpy as np
import pytest

import dllm_inputs as I
import oracle as O

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

TINY = O.OracleConfig()


@pytest.fixture(scope="module")
def model():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    import paper_2606_13740_gb300 as pkg
    pkg.lib()
    return O.Model(TINY)


def _gpu_ctx(max_ctx=256, max_window=160, max_batch=1):
    from paper_2606_13740_gb300 import Config, Context
    return Context(Config(max_ctx=max_ctx, max_window=max_window, max_batch=max_batch))


def test_weights_bit_exact(model):
    ctx = _gpu_ctx()
    for which, tid in ((1, O.T_EMBED), (2, O.T_HEAD)):
        assert np.array_equal(ctx.dllm_get_weight(-1, which), model.weight(-1, tid))
    for layer in range(TINY.n_layers):
        for w in range(7):
            assert np.array_equal(ctx.dllm_get_weight(layer, w), model.weight(layer, w)), (layer, w)
    ctx.close()


def _unambiguous_commits(od, o_tok_before, o_st_before, c0, c1, w0, k):
    masked = [p for p in range(c0, c1) if o_st_before[p] == O.MASKED]
    if k == 0 or k >= len(masked):
        return True
    c = sorted((float(od["conf"][p - w0]) for p in masked), reverse=True)
    return (c[k - 1] - c[k]) > 0.02 * c[k - 1]


def _run_teacher_forced(model, osched, gsched, prompt, gen_len, ctx, check=None):
    sess = O.Session(model, osched, prompt, gen_len)
    sess.prefill()
    ctx.dllm_prefill(gsched, prompt, gen_len)
    ctx.dllm_set_debug(1)
    steps = 0
    worst = 0.0
    while True:
        o_more = sess.begin_block()
        g_more = ctx.dllm_begin_block()
        assert o_more == g_more
        if not o_more:
            break
        while True:
            o_tok0, o_st0, _ = sess.state()
            g_tok0, g_st0, _ = ctx.dllm_get_state()
            assert np.array_equal(g_tok0[0], o_tok0) and np.array_equal(g_st0[0], o_st0)
            oo = sess.step(keep_logits=True)
            go = ctx.dllm_denoise_step()
            ow, gw = sess.window(), ctx.dllm_window()
            for key in ("w0", "T", "c0", "c1", "kv_len", "spec_on", "step"):
                assert ow[key] == gw[key], (key, ow, gw)
            od = sess.decisions(logits=True)
            gd = ctx.dllm_get_step_debug(logits=True)
            lg, ref = gd["logits"][0], od["logits"]
            rel = float(np.linalg.norm(lg - ref) / np.linalg.norm(ref))
            worst = max(worst, rel)
            assert rel <= 1e-2, rel
            safe = od["margin"] > 0.05
            assert np.array_equal(gd["x0"][0][safe], od["x0"][safe])
            assert not (gd["x0"][0] == TINY.mask_id).any()
            assert np.allclose(gd["conf"][0], od["conf"], rtol=0.05)
            for key in ("n_committed", "n_drafts", "block_done", "masked_after"):
                assert go[key] == oo[key], (key, go, oo)
            g_tok, g_st, _ = ctx.dllm_get_state()
            o_tok, o_st, _ = sess.state()
            if check is not None:
                check(sess, ctx, oo, go, (o_tok0, o_st0), (o_tok, o_st), (g_tok[0], g_st[0]))
            if _unambiguous_commits(od, o_tok0, o_st0, ow["c0"], ow["c1"], ow["w0"], oo["n_committed"]):
                newly_o = (o_st == O.COMMITTED) & (o_st0 == O.MASKED)
                newly_g = (g_st[0] == O.COMMITTED) & (g_st0[0] == O.MASKED)
                assert np.array_equal(newly_o, newly_g)
            ctx.dllm_set_state(o_tok[None], o_st[None])  # teacher forcing
            steps += 1
            if oo["block_done"]:
                break
    o_tok, o_st, o_kv = sess.state()
    g_tok, g_st, g_kv = ctx.dllm_get_state()
    assert g_kv[0] == o_kv
    assert np.array_equal(g_tok[0], o_tok) and np.array_equal(g_st[0], o_st)
    return sess, steps, worst


def test_blockwise_prefix_cache_teacher_forced(model):
    """Tiny config: 64-token prompt, 2 blocks of 32, 8 steps/block (4 commits/step)."""
    from paper_2606_13740_gb300 import Sched
    prompt = I.uniform_prompt(64, TINY.vocab, TINY.mask_id)
    ctx = _gpu_ctx()
    sess, steps, worst = _run_teacher_forced(model, O.OracleSched(steps_per_block=8), Sched(steps_per_block=8),
                                             prompt, 64, ctx)
    assert steps == 16
    kv_len = sess.state()[2]
    for layer in range(TINY.n_layers):
        for which in (0, 1):
            ref = sess.prefix_kv(layer, which)
            got = ctx.dllm_get_kv(layer, which, 0, 0, kv_len)
            assert np.linalg.norm(got - ref) / np.linalg.norm(ref) <= 1e-2
    ctx.close()


def test_vanilla_full_sequence_teacher_forced(model):
    from paper_2606_13740_gb300 import Sched
    prompt = I.uniform_prompt(16, TINY.vocab, TINY.mask_id, seed=11)
    ctx = _gpu_ctx()
    _, steps, _ = _run_teacher_forced(model, O.OracleSched(steps_per_block=8, use_prefix_cache=0),
                                      Sched(steps_per_block=8, use_prefix_cache=0), prompt, 32, ctx)
    assert steps == 8
    ctx.close()


def test_speculative_revision_teacher_forced(model):
    """Lookahead of 2 blocks at <= 8 masked, re-mask below 0.5 (config-4 rules)."""
    from paper_2606_13740_gb300 import Sched
    prompt = I.uniform_prompt(32, TINY.vocab, TINY.mask_id, seed=22)
    osched = O.OracleSched(steps_per_block=16, spec_blocks=2, spec_trigger=8, theta_remask=0.5, remask_max=1)
    gsched = Sched(steps_per_block=16, spec_blocks=2, spec_trigger=8, theta_remask=0.5, remask_max=1)
    ctx = _gpu_ctx()
    _, steps, _ = _run_teacher_forced(model, osched, gsched, prompt, 128, ctx)
    assert steps >= 4 * 1
    ctx.close()


@pytest.mark.parametrize("theta_visible,steps_per_block", [(2.0, 32), (0.0, 1)])
def test_threshold_commit_teacher_forced(model, theta_visible, steps_per_block):
    """Staged token stabilization at its two exact ends: theta_visible out of reach (the
    fallback, one position per step, 32 steps per block) and 0 (the whole block at once)."""
    from paper_2606_13740_gb300 import COMMIT_THRESHOLD, Sched
    prompt = I.uniform_prompt(32, TINY.vocab, TINY.mask_id, seed=41)
    osched = O.OracleSched(steps_per_block=8, commit_mode=1, theta_visible=theta_visible, theta_stable=2.0)
    gsched = Sched(steps_per_block=8, commit_mode=COMMIT_THRESHOLD, theta_visible=theta_visible, theta_stable=2.0)
    ctx = _gpu_ctx()
    _, steps, _ = _run_teacher_forced(model, osched, gsched, prompt, 64, ctx)
    assert steps == 2 * steps_per_block
    ctx.close()


def test_threshold_commit_generation_mid_thresholds(model):
    """Thresholds inside the tiny model's confidence range: every step commits at least one
    position, positions reaching theta_stable go straight to STABLE, every block finishes in
    at most 32 steps, and a rerun gives the same tokens."""
    from paper_2606_13740_gb300 import COMMIT_THRESHOLD, STABLE, Sched
    prompt = I.uniform_prompt(32, TINY.vocab, TINY.mask_id, seed=42)
    sched = Sched(steps_per_block=8, commit_mode=COMMIT_THRESHOLD, theta_visible=0.00256, theta_stable=0.0026)
    ctx = _gpu_ctx()
    ctx.dllm_prefill(sched, prompt, 64)
    blocks, steps, stable_direct = 0, 0, 0
    while ctx.dllm_begin_block():
        n = 0
        while True:
            out = ctx.dllm_denoise_step()
            n += 1
            assert out["n_committed"] >= 1
            stable_direct += out["n_stable"]
            if out["block_done"]:
                break
        assert 1 <= n <= 32
        blocks += 1
        steps += n
    tok, st, kv = ctx.dllm_get_state()
    assert blocks == 2 and kv[0] == 96 and not (tok[0, 32:96] == TINY.mask_id).any()
    assert stable_direct == int((st[0, 32:96] == STABLE).sum())
    again, _ = ctx.dllm_generate(sched, prompt, 64)
    assert np.array_equal(again[0], tok[0, 32:96])
    ctx.close()


@pytest.mark.parametrize("theta_stable", [2.0, 0.0])
def test_sparse_cache_refresh_teacher_forced(model, theta_stable):
    """Sparse cache refresh of 8 visible prefix positions per step (Sec. 3.3).  Every step: the
    same tracked positions as the oracle, their decisions within tolerance, the same refresh and
    stabilization counts, and the same prefix states after the step; at the end the prefix K/V
    (refreshed in place by the merges) against the oracle's.  theta_stable 2: the rows only
    refresh; 0: every tracked row also becomes STABLE."""
    from paper_2606_13740_gb300 import Sched
    prompt = I.uniform_prompt(32, TINY.vocab, TINY.mask_id, seed=61)
    osched = O.OracleSched(steps_per_block=4, scr_rows=8, theta_stable=theta_stable)
    gsched = Sched(steps_per_block=4, scr_rows=8, theta_stable=theta_stable)
    counts = {"steps_with_rows": 0}

    def check(sess, ctx, oo, go, before, o_after, g_after):
        od, gd = sess.scr_decisions(), ctx.dllm_get_scr_debug()
        n = len(od["pos"])
        assert np.array_equal(gd["pos"][:n], od["pos"]) and (gd["pos"][n:] == -1).all()
        if n:
            counts["steps_with_rows"] += 1
            assert np.allclose(gd["conf"][:n], od["conf"], rtol=0.05)
            assert np.allclose(gd["tokconf"][:n], od["tokconf"], rtol=0.05)
            safe = od["margin"] > 0.05
            assert np.array_equal(gd["x0"][:n][safe], od["x0"][safe])
        for key in ("n_refreshed", "n_revised", "n_stable"):
            assert go[key] == oo[key], (key, go, oo)
        kv = sess.window()["kv_len"]
        assert np.array_equal(g_after[1][:kv], o_after[1][:kv])  # the prefix states
        assert np.array_equal(g_after[0][:kv], o_after[0][:kv])

    ctx = _gpu_ctx()
    sess, steps, worst = _run_teacher_forced(model, osched, gsched, prompt, 96, ctx, check)
    assert steps == 12 and counts["steps_with_rows"] >= 4
    kv_len = sess.state()[2]
    for layer in range(TINY.n_layers):
        for which in (0, 1):
            ref = sess.prefix_kv(layer, which)
            got = ctx.dllm_get_kv(layer, which, 0, 0, kv_len)
            assert np.linalg.norm(got - ref) / np.linalg.norm(ref) <= 1e-2
    ctx.close()


def test_adaptive_lookahead_teacher_forced(model):
    """Adaptive lookahead (Sec. 3.2) from a latency table: every step's window equals the
    oracle's (the harness compares them), and the table admits two future blocks, not three."""
    from paper_2606_13740_gb300 import Sched
    prompt = I.uniform_prompt(32, TINY.vocab, TINY.mask_id, seed=71)
    lat = (1.0, 1.05, 1.1, 2.0)
    osched = O.OracleSched(steps_per_block=8, spec_blocks=3, spec_trigger=4, spec_allowance=0.12, spec_lat=lat)
    gsched = Sched(steps_per_block=8, spec_blocks=3, spec_trigger=4, spec_allowance=0.12, spec_lat=lat)
    ctx = _gpu_ctx(max_window=160)
    windows = []

    def check(sess, ctx, oo, go, before, o_after, g_after):
        windows.append(sess.window()["T"])

    _run_teacher_forced(model, osched, gsched, prompt, 160, ctx, check)
    assert 96 in windows and 128 not in windows
    ctx.close()


def test_sparse_cache_refresh_batch_matches_single_sequences(model):
    """Two sequences with sparse cache refresh: each one's tokens, states, per-step refresh
    counts and refreshed prefix K/V are bit-identical to its own single-sequence run.  (32
    refresh rows: a sequence's rows stay a multiple of the epilogue's 32-token chunks, so its
    RoPE takes the same path whatever the batch.)"""
    from paper_2606_13740_gb300 import Sched
    prompts = I.uniform_prompt(32, TINY.vocab, TINY.mask_id, batch=2, seed=81)
    sched = Sched(steps_per_block=4, scr_rows=32, theta_stable=0.0015, theta_remask=0.0023, remask_max=1)

    def run(p):
        ctx = _gpu_ctx(max_batch=2, max_window=64)
        ctx.dllm_prefill(sched, p, 96)
        counts = []
        while ctx.dllm_begin_block():
            while True:
                out = ctx.dllm_denoise_step()
                counts.append((out["n_refreshed"], out["n_revised"], out["n_stable"]))
                if out["block_done"]:
                    break
        tok, st, kv = ctx.dllm_get_state()
        kvs = [[ctx.dllm_get_kv(l, w, b, 0, int(kv[b])) for l in range(TINY.n_layers) for w in (0, 1)]
               for b in range(p.shape[0])]
        ctx.close()
        return tok, st, counts, kvs

    tok2, st2, c2, kv2 = run(prompts)
    for b in range(2):
        tok1, st1, c1, kv1 = run(prompts[b:b + 1])
        assert np.array_equal(tok2[b], tok1[0]) and np.array_equal(st2[b], st1[0])
        for x, y in zip(kv2[b], kv1[0]):
            assert np.array_equal(x, y)
        if b == 0:
            single0 = c1
        else:
            summed = [tuple(p + q for p, q in zip(u, v)) for u, v in zip(single0, c1)]
            assert c2 == summed
    assert sum(c[0] for c in c2) > 0


def test_generate_matches_stepwise_and_is_deterministic(model):
    from paper_2606_13740_gb300 import Sched
    prompt = I.uniform_prompt(64, TINY.vocab, TINY.mask_id)
    ctx = _gpu_ctx()
    a, stats = ctx.dllm_generate(Sched(steps_per_block=8), prompt, 64)
    b, _ = ctx.dllm_generate(Sched(steps_per_block=8), prompt, 64)
    assert np.array_equal(a, b)
    assert stats == {"steps": 16, "spec_steps": 0, "blocks": 2}
    assert not (a == TINY.mask_id).any()
    ctx.close()


def test_batch_sequences_are_independent(model):
    from paper_2606_13740_gb300 import Sched
    prompts = I.uniform_prompt(32, TINY.vocab, TINY.mask_id, batch=3, seed=5)
    ctx = _gpu_ctx(max_batch=3, max_window=64)
    batched, _ = ctx.dllm_generate(Sched(steps_per_block=8), prompts, 64)
    for b in range(3):
        single, _ = ctx.dllm_generate(Sched(steps_per_block=8), prompts[b:b + 1], 64)
        assert np.array_equal(single[0], batched[b])
    ctx.close()


def test_rewind_repeats_identical_step(model):
    from paper_2606_13740_gb300 import Sched
    prompt = I.uniform_prompt(64, TINY.vocab, TINY.mask_id)
    ctx = _gpu_ctx()
    ctx.dllm_prefill(Sched(steps_per_block=8), prompt, 32)
    ctx.dllm_begin_block()
    ctx.dllm_denoise_step()
    s1 = ctx.dllm_get_state()
    ctx.dllm_rewind_block()
    ctx.dllm_denoise_step()
    s2 = ctx.dllm_get_state()
    assert np.array_equal(s1[0], s2[0]) and np.array_equal(s1[1], s2[1])
    ctx.close()


def test_errors_poison_context(model):
    """Argument and capacity errors leave the context usable; a device-side failure (here a
    bounded wait that runs out) poisons it: the call reports DLLM_ETIMEOUT, every later call
    DLLM_ESTATE, and a fresh context works."""
    from paper_2606_13740_gb300 import DllmError, Sched
    ctx = _gpu_ctx(max_ctx=96)
    with pytest.raises(DllmError) as e:  # capacity
        ctx.dllm_prefill(Sched(), I.uniform_prompt(64, TINY.vocab, TINY.mask_id), 64)
    assert e.value.code == -6
    with pytest.raises(DllmError) as e:  # no request yet
        ctx.dllm_begin_block()
    assert e.value.code == -1
    bad = I.uniform_prompt(32, TINY.vocab, TINY.mask_id)
    bad[5] = TINY.vocab  # an id out of range: rejected before the request starts
    with pytest.raises(DllmError) as e:
        ctx.dllm_prefill(Sched(steps_per_block=8), bad, 32)
    assert e.value.code == -1
    prompt = I.uniform_prompt(32, TINY.vocab, TINY.mask_id)
    ctx.dllm_prefill(Sched(steps_per_block=8), prompt, 32)
    ctx.dllm_begin_block()
    ctx.dllm_denoise_step()
    with pytest.raises(DllmError) as e:  # block unfinished
        ctx.dllm_begin_block()
    assert e.value.code == -1
    out = ctx.dllm_denoise_step()  # still usable
    assert out["n_committed"] == 4
    ctx.dllm_set_debug(32)  # the next step's first projection waits for a word nothing writes
    with pytest.raises(DllmError) as e:
        ctx.dllm_denoise_step()
    assert e.value.code == -4  # DLLM_ETIMEOUT
    for call in (ctx.dllm_denoise_step, ctx.dllm_begin_block, ctx.dllm_get_state, ctx.dllm_sync):
        with pytest.raises(DllmError) as e:
            call()
        assert e.value.code == -5  # DLLM_ESTATE: poisoned
    ctx.close()
    fresh = _gpu_ctx(max_ctx=96)
    fresh.dllm_prefill(Sched(steps_per_block=8), prompt, 32)
    fresh.dllm_begin_block()
    assert fresh.dllm_denoise_step()["n_committed"] == 4
    fresh.close()


@pytest.mark.parametrize("slide", [0, 1])
def test_selective_logits_skipping_teacher_forced(model, slide):
    """Selective logits skipping (Sec. 3.3) against the oracle, which decides every row: each
    step, the rows whose position is MASKED, COMMITTED or DRAFT carry the oracle's decisions,
    STABLE rows carry none (x0 -1, conf and tokconf 0), and the commit bookkeeping is that of
    the oracle.  Revision and one lookahead block run; between steps, teacher forcing makes
    every other visible position STABLE in both (the thresholds stay out of the tiny model's
    confidence range, so no decision sits on one of them)."""
    from paper_2606_13740_gb300 import Sched
    prompt = I.uniform_prompt(32, TINY.vocab, TINY.mask_id, seed=43)
    kw = dict(steps_per_block=8, theta_remask=0.5, remask_max=1, spec_blocks=1, spec_trigger=16, slide=slide)
    sess = O.Session(model, O.OracleSched(**kw), prompt, 96)
    sess.prefill()
    ctx = _gpu_ctx()
    ctx.dllm_prefill(Sched(sls=1, **kw), prompt, 96)
    skipped, needed, states = 0, 0, set()
    while True:
        more = sess.begin_block()
        assert more == ctx.dllm_begin_block()
        if not more:
            break
        while True:
            o_tok0, o_st0, _ = sess.state()
            g_tok0, g_st0, _ = ctx.dllm_get_state()
            assert np.array_equal(g_tok0[0], o_tok0) and np.array_equal(g_st0[0], o_st0)
            oo = sess.step()
            go = ctx.dllm_denoise_step()
            ow, gw = sess.window(), ctx.dllm_window()
            for key in ("w0", "T", "c0", "c1", "kv_len", "spec_on", "step"):
                assert ow[key] == gw[key], (key, ow, gw)
            od = sess.decisions()
            gd = ctx.dllm_get_step_debug()
            w0, T = ow["w0"], ow["T"]
            win = o_st0[w0:w0 + T]
            states.update(int(s) for s in win)
            need = np.isin(win, (O.MASKED, O.COMMITTED, O.DRAFT))
            gx, gc, gt = gd["x0"][0], gd["conf"][0], gd["tokconf"][0]
            assert (gx[~need] == -1).all() and (gc[~need] == 0).all() and (gt[~need] == 0).all()
            safe = need & (od["margin"] > 0.05)
            assert np.array_equal(gx[safe], od["x0"][safe])
            assert np.allclose(gc[need], od["conf"][need], rtol=0.05)
            assert np.allclose(gt[need], od["tokconf"][need], rtol=0.05, atol=1e-7)
            for key in ("n_committed", "n_remasked", "n_stable", "n_drafts", "block_done", "masked_after"):
                assert go[key] == oo[key], (key, go, oo)
            skipped += int((~need).sum())
            needed += int(need.sum())
            o_tok, o_st, _ = sess.state()
            vis = np.flatnonzero(o_st == O.COMMITTED)
            o_st[vis[::2]] = O.STABLE
            sess.set_state(o_tok, o_st)
            ctx.dllm_set_state(o_tok[None], o_st[None])  # teacher forcing
            if oo["block_done"]:
                break
    assert skipped > 0 and needed > 0
    assert {O.MASKED, O.COMMITTED, O.STABLE, O.DRAFT} <= states
    ctx.close()


@pytest.mark.parametrize("n_stable", [0, 24, 32])
def test_selective_logits_skipping_batch_one_step(model, n_stable):
    """Sixteen sequences, one step over their 32-token blocks (two 256-token head tiles without
    skipping): sequence b has max(0, n_stable - 2 b) of its block positions STABLE and a third
    of the rest visible.  With n_stable = 32 sequence 0 needs no row and the needed rows fit
    one token tile; with 24 they end inside the second tile.  Every needed row's decision
    matches the oracle's for that sequence and state; every other row carries none."""
    from paper_2606_13740_gb300 import Sched
    B, gen = 16, 64
    prompts = I.uniform_prompt(32, TINY.vocab, TINY.mask_id, batch=B, seed=90)
    kw = dict(steps_per_block=8, theta_remask=0.5, remask_max=1)
    ctx = _gpu_ctx(max_batch=B, max_window=64)
    ctx.dllm_prefill(Sched(sls=1, **kw), prompts, gen)
    assert ctx.dllm_begin_block()
    tok, st, kv = ctx.dllm_get_state()
    rng = np.random.default_rng(91)
    for b in range(B):
        w0 = int(kv[b])
        k = max(0, n_stable - 2 * b)
        pos = w0 + rng.permutation(32)
        tok[b, pos[:k]] = rng.integers(0, TINY.mask_id, k)
        st[b, pos[:k]] = O.STABLE
        vis = pos[k:k + (32 - k) // 3]
        tok[b, vis] = rng.integers(0, TINY.mask_id, len(vis))
        st[b, vis] = O.COMMITTED
    ctx.dllm_set_state(tok, st)
    ctx.dllm_denoise_step()
    assert ctx.dllm_window()["T"] == 32
    gd = ctx.dllm_get_step_debug()
    n_need = []
    for b in range(B):
        sess = O.Session(model, O.OracleSched(**kw), prompts[b], gen)
        sess.prefill()
        assert sess.begin_block()
        sess.set_state(tok[b], st[b])
        sess.step()
        assert sess.window()["T"] == 32
        od = sess.decisions()
        win = st[b, int(kv[b]):int(kv[b]) + 32]
        need = np.isin(win, (O.MASKED, O.COMMITTED, O.DRAFT))
        n_need.append(int(need.sum()))
        gx, gc = gd["x0"][b], gd["conf"][b]
        assert (gx[~need] == -1).all() and (gc[~need] == 0).all()
        safe = need & (od["margin"] > 0.05)
        assert np.array_equal(gx[safe], od["x0"][safe])
        assert np.allclose(gc[need], od["conf"][need], rtol=0.05)
    if n_stable == 32:
        assert n_need[0] == 0 and sum(n_need) <= 256
    elif n_stable == 24:
        assert 256 < sum(n_need) < 512
    ctx.close()


@pytest.mark.parametrize("spec", [0, 1])
def test_continuous_sliding_teacher_forced(model, spec):
    """Continuous sliding (Sec. 3.2) against the oracle: every step's window (start, size, cache
    frontier), decisions and bookkeeping, the final ids, states and cache; the window does move
    past its block start, with and without a lookahead block."""
    from paper_2606_13740_gb300 import Sched
    prompt = I.uniform_prompt(32, TINY.vocab, TINY.mask_id, seed=62)
    kw = dict(steps_per_block=8, slide=1, spec_blocks=spec, spec_trigger=8)
    ctx = _gpu_ctx()
    moved = []

    def check(sess, ctx_, oo, go, pre_o, post_o, post_g):
        w = sess.window()
        moved.append(w["kv_len"] > w["c0"])

    sess, steps, _ = _run_teacher_forced(model, O.OracleSched(**kw), Sched(**kw), prompt, 96, ctx, check=check)
    assert any(moved)
    kv_len = sess.state()[2]
    for layer in range(TINY.n_layers):
        for which in (0, 1):
            ref = sess.prefix_kv(layer, which)
            got = ctx.dllm_get_kv(layer, which, 0, 0, kv_len)
            assert np.linalg.norm(got - ref) / np.linalg.norm(ref) <= 1e-2
    ctx.close()


@pytest.mark.parametrize("case", ["refresh", "threshold_fallback"])
def test_continuous_sliding_with_other_rows(model, case):
    """Continuous sliding combined with sparse cache refresh (slid positions are COMMITTED
    prefix positions, so they become refresh rows) and with the threshold commit's one-position
    fallback, teacher-forced against the oracle."""
    from paper_2606_13740_gb300 import COMMIT_THRESHOLD, Sched
    prompt = I.uniform_prompt(32, TINY.vocab, TINY.mask_id, seed=63)
    if case == "refresh":
        okw = gkw = dict(steps_per_block=8, slide=1, scr_rows=8, theta_stable=2.0)
    else:
        okw = dict(steps_per_block=8, slide=1, commit_mode=1, theta_visible=2.0, theta_stable=2.0)
        gkw = dict(okw, commit_mode=COMMIT_THRESHOLD)
    ctx = _gpu_ctx()
    moved = []

    def check(sess, ctx_, oo, go, pre_o, post_o, post_g):
        w = sess.window()
        moved.append(w["kv_len"] > w["c0"])
        assert go["n_refreshed"] == oo["n_refreshed"] and go["n_revised"] == oo["n_revised"]

    _run_teacher_forced(model, O.OracleSched(**okw), Sched(**gkw), prompt, 64, ctx, check=check)
    assert any(moved)
    ctx.close()


def test_new_request_takes_its_own_schedule(model):
    """The captured step bakes in the schedule's commit rule: a new request on the same context
    (same window, batch and cache length) must run under its own schedule, not replay the last
    one's step."""
    from paper_2606_13740_gb300 import COMMIT_THRESHOLD, Sched
    prompt = I.uniform_prompt(32, TINY.vocab, TINY.mask_id, seed=64)
    ctx = _gpu_ctx()
    _, s1 = ctx.dllm_generate(Sched(steps_per_block=8), prompt, 64)
    _, s2 = ctx.dllm_generate(Sched(steps_per_block=8, commit_mode=COMMIT_THRESHOLD, theta_visible=0.0), prompt, 64)
    _, s3 = ctx.dllm_generate(Sched(steps_per_block=8), prompt, 64)
    assert s1["steps"] == s3["steps"] == 16
    assert s2["steps"] == 2  # a whole block per step
    ctx.close()
