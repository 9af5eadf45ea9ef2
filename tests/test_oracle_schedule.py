"""Pins of the oracle's decoding loop: the commit schedule, top-k selection,
re-masking, drafts, prefix-KV bookkeeping, and equivalence with a separately
written vanilla LLaDA sampler (Sec. 2.1, Sec. 3.2, Sec. 3.3 of the paper).
"""
import numpy as np
import pytest

import dllm_inputs as I
import oracle as O

TINY = O.OracleConfig()  # 2 layers, d 256, 4x64 heads, ffn 688, vocab 1024, mask 1023


@pytest.fixture(scope="module")
def tiny_model(oracle_lib):
    return O.Model(TINY)


def _llada_schedule(m0, S):
    """LLaDA's front-loaded per-step transfer counts (closed form)."""
    base, rem = divmod(m0, S)
    return [base + (1 if s < rem else 0) for s in range(S)]


# ------------------------------------------------------------ commit pass
@pytest.mark.parametrize("m0,S", [(32, 8), (32, 32), (24, 32), (5, 4), (1, 3), (31, 7)])
def test_commit_counts_follow_llada_closed_form(oracle_lib, m0, S):
    n = 40
    tok = np.full(n, TINY.mask_id, np.int32)
    st = np.full(n, O.MASKED, np.uint8)
    c0, c1 = 4, 4 + 32
    st[:c0] = O.FIXED
    st[c0:c1][m0:] = O.COMMITTED  # 32 - m0 already committed
    tok[:c0] = 5
    tok[c0:c1][m0:] = 6
    sched = O.OracleSched(steps_per_block=S, block_len=32)
    got = []
    for s in range(S):
        conf = I.scripted_confidences(n, seed=100 + s)
        x0 = np.arange(n, dtype=np.int32) % 1000
        tok, st, out = O.commit(sched, TINY.mask_id, tok, st, 0, n, c0, c1, s, x0, conf, np.zeros(n, np.float32))
        got.append(out["n_committed"])
        assert out["masked_after"] == int((st[c0:c1] == O.MASKED).sum())
    assert got == _llada_schedule(m0, S)
    assert sum(got) == m0
    assert not (st[c0:c1] == O.MASKED).any()
    assert not (tok[c0:c1] == TINY.mask_id).any()


@pytest.mark.parametrize("seed", range(6))
def test_commit_selects_top_k_by_confidence_then_position(oracle_lib, seed):
    n, c0, c1 = 48, 8, 40
    rng = np.random.default_rng(seed)
    st = np.where(rng.random(n) < 0.6, O.MASKED, O.COMMITTED).astype(np.uint8)
    tok = np.where(st == O.MASKED, TINY.mask_id, 1).astype(np.int32)
    conf = I.scripted_confidences(n, seed=seed, ties=True)
    x0 = rng.integers(0, 1000, n).astype(np.int32)
    S, s = 8, 3
    sched = O.OracleSched(steps_per_block=S)
    tok2, st2, out = O.commit(sched, TINY.mask_id, tok, st, 0, n, c0, c1, s, x0, conf, np.zeros(n, np.float32))
    masked = [p for p in range(c0, c1) if st[p] == O.MASKED]
    k = -(-len(masked) // (S - s)) if masked else 0
    want = sorted(masked, key=lambda p: (-conf[p], p))[:k]
    got = [p for p in range(n) if st2[p] != st[p]]
    assert sorted(want) == got
    assert out["n_committed"] == k
    assert all(tok2[p] == x0[p] and st2[p] == O.COMMITTED for p in want)
    outside = [p for p in range(n) if not (c0 <= p < c1)]
    assert np.array_equal(tok2[outside], tok[outside])


def test_remask_lowest_confidence_and_stable_promotion(oracle_lib):
    n, c0, c1 = 32, 0, 32
    st = np.full(n, O.COMMITTED, np.uint8)
    st[20:] = O.MASKED
    tok = np.where(st == O.MASKED, TINY.mask_id, 3).astype(np.int32)
    tokconf = np.full(n, 0.6, np.float32)
    tokconf[[2, 5, 9]] = [0.3, 0.1, 0.1]  # below 0.5: 5 and 9 tie, 5 wins
    tokconf[[1, 4]] = [0.95, 0.9]  # at or above theta_stable
    conf = I.scripted_confidences(n, seed=7)
    x0 = np.full(n, 11, np.int32)
    sched = O.OracleSched(steps_per_block=16, theta_remask=0.5, theta_stable=0.9, remask_max=1)
    tok2, st2, out = O.commit(sched, TINY.mask_id, tok, st, 0, n, c0, c1, 2, x0, conf, tokconf)
    assert out["n_remasked"] == 1 and out["n_stable"] == 2
    assert st2[1] == O.STABLE and st2[4] == O.STABLE
    # position 5 was re-masked; it competes with the other masked positions
    masked_before_commit = sorted([5] + list(range(20, 32)))
    k = -(-len(masked_before_commit) // (16 - 2))
    chosen = sorted(masked_before_commit, key=lambda p: (-conf[p], p))[:k]
    for p in masked_before_commit:
        if p in chosen:
            assert st2[p] == O.COMMITTED and tok2[p] == 11
        else:
            assert st2[p] == O.MASKED and tok2[p] == TINY.mask_id
    assert st2[9] == O.COMMITTED and tok2[9] == 3 and st2[2] == O.COMMITTED
    # two re-masks allowed: both ties at 0.1 go
    sched2 = O.OracleSched(steps_per_block=16, theta_remask=0.5, remask_max=2)
    conf2 = np.ones(n, np.float32)
    conf2[[5, 9]] = 0.0  # the re-masked positions lose the commit pass
    _, st3, out3 = O.commit(sched2, TINY.mask_id, tok, st, 0, n, c0, c1, 2, x0, conf2, tokconf)
    assert out3["n_remasked"] == 2 and st3[5] == O.MASKED and st3[9] == O.MASKED and st3[2] == O.COMMITTED


def test_revision_disabled_on_last_step_and_at_zero_threshold(oracle_lib):
    n = 32
    st = np.full(n, O.COMMITTED, np.uint8)
    st[-1] = O.MASKED
    tok = np.where(st == O.MASKED, TINY.mask_id, 3).astype(np.int32)
    tokconf = np.full(n, 0.01, np.float32)
    x0 = np.full(n, 4, np.int32)
    conf = np.ones(n, np.float32)
    last = O.OracleSched(steps_per_block=8, theta_remask=0.5)
    _, st2, out = O.commit(last, TINY.mask_id, tok, st, 0, n, 0, n, 7, x0, conf, tokconf)
    assert out["n_remasked"] == 0 and out["block_done"] == 1
    off = O.OracleSched(steps_per_block=8, theta_remask=0.0)
    _, _, out = O.commit(off, TINY.mask_id, tok, st, 0, n, 0, n, 2, x0, conf, tokconf)
    assert out["n_remasked"] == 0 and out["n_stable"] == 0


def test_drafts_one_per_speculative_block(oracle_lib):
    n, bl = 128, 32
    c0, c1 = 32, 64
    st = np.full(n, O.MASKED, np.uint8)
    st[:c0] = O.FIXED
    st[c0:c0 + 28] = O.COMMITTED
    st[64 + 3] = O.DRAFT
    tok = np.where(st == O.MASKED, TINY.mask_id, 2).astype(np.int32)
    conf = I.scripted_confidences(n, seed=9, ties=True)
    x0 = (np.arange(n) % 900).astype(np.int32)
    sched = O.OracleSched(steps_per_block=32, spec_blocks=2, spec_trigger=8, use_prefix_cache=1)
    w0, T = c0, 96  # decisions are indexed by window offset
    tok2, st2, out = O.commit(sched, TINY.mask_id, tok, st, w0, T, c0, c1, 5, x0[w0:w0 + T], conf[w0:w0 + T],
                              np.zeros(T, np.float32))
    assert out["n_drafts"] == 2
    for b0, b1 in ((64, 96), (96, 128)):
        new = [p for p in range(b0, b1) if st2[p] == O.DRAFT and st[p] != O.DRAFT]
        cand = [p for p in range(b0, b1) if st[p] == O.MASKED]
        assert new == [sorted(cand, key=lambda p: (-conf[p], p))[0]]
        assert tok2[new[0]] == x0[new[0]]


# ------------------------------------------------------------ sessions
def _vanilla_llada(model, prompt, gen_len, block_len, steps_per_block):
    """Separately written LLaDA sampler: full sequence every step, the
    front-loaded per-block transfer schedule, top-k by confidence."""
    cfg = model.cfg
    Lp = prompt.size
    x = np.concatenate([prompt, np.full(gen_len, cfg.mask_id, np.int32)])
    pos = np.arange(x.size, dtype=np.int32)
    for b in range(gen_len // block_len):
        lo, hi = Lp + b * block_len, Lp + (b + 1) * block_len
        counts = _llada_schedule(int((x[lo:hi] == cfg.mask_id).sum()), steps_per_block)
        for s in range(steps_per_block):
            logits = O.forward(model, x, pos)["logits"]
            dec = [O.decide(logits[p], cfg.mask_id, x[p]) for p in range(x.size)]
            masked = [p for p in range(lo, hi) if x[p] == cfg.mask_id]
            chosen = sorted(masked, key=lambda p: (-dec[p][1], p))[:counts[s]]
            for p in chosen:
                x[p] = dec[p][0]
    return x[Lp:]


def test_vanilla_equivalence(tiny_model):
    """Cache off and one block spanning the whole generation equals the
    vanilla full-sequence sampler."""
    prompt = I.uniform_prompt(16, TINY.vocab, TINY.mask_id, seed=11)
    gen = 32
    want = _vanilla_llada(tiny_model, prompt, gen, gen, 8)
    sess = O.Session(tiny_model, O.OracleSched(steps_per_block=8, block_len=gen, use_prefix_cache=0), prompt, gen)
    got = sess.generate()
    assert np.array_equal(got, want)


def test_cache_off_blockwise_equals_semi_autoregressive_llada(tiny_model):
    prompt = I.uniform_prompt(8, TINY.vocab, TINY.mask_id, seed=12)
    want = _vanilla_llada(tiny_model, prompt, 64, 32, 4)
    sess = O.Session(tiny_model, O.OracleSched(steps_per_block=4, block_len=32, use_prefix_cache=0), prompt, 64)
    assert np.array_equal(sess.generate(), want)


def test_incremental_prefix_kv_equals_block_causal_recompute(tiny_model):
    prompt = I.uniform_prompt(40, TINY.vocab, TINY.mask_id, seed=13)
    sess = O.Session(tiny_model, O.OracleSched(steps_per_block=8), prompt, 64)
    gen = sess.generate()
    tok, st, kv_len = sess.state()
    assert kv_len == 40 + 64
    assert (st[40:] == O.COMMITTED).all() and np.array_equal(tok[40:], gen)
    group = np.array([0] * 40 + [1] * 32 + [2] * 32, np.int32)
    full = O.forward(tiny_model, tok, np.arange(tok.size), group=group, want_kv=True, logits=False)
    for layer in range(TINY.n_layers):
        assert np.array_equal(sess.prefix_kv(layer, 0), full["k"][layer])
        assert np.array_equal(sess.prefix_kv(layer, 1), full["v"][layer])


def test_session_schedule_and_mask_invariants(tiny_model):
    prompt = I.uniform_prompt(64, TINY.vocab, TINY.mask_id)
    sess = O.Session(tiny_model, O.OracleSched(steps_per_block=8), prompt, 64)
    sess.prefill()
    blocks = 0
    while sess.begin_block():
        counts = []
        while True:
            w = sess.window()
            out = sess.step()
            counts.append(out["n_committed"])
            assert sess.window()["T"] == 32 and sess.window()["w0"] == 64 + 32 * blocks
            if out["block_done"]:
                break
        assert counts == [4] * 8
        assert sess.state()[2] == 64 + 32 * blocks
        blocks += 1
    tok, st, kv = sess.state()
    assert blocks == 2 and kv == 128
    assert not (tok[64:] == TINY.mask_id).any()


def test_speculation_trigger_off_equals_plain_blocks(tiny_model):
    prompt = I.uniform_prompt(32, TINY.vocab, TINY.mask_id, seed=21)
    plain = O.Session(tiny_model, O.OracleSched(steps_per_block=16), prompt, 96).generate()
    never = O.Session(tiny_model, O.OracleSched(steps_per_block=16, spec_blocks=2, spec_trigger=-1), prompt, 96)
    assert np.array_equal(never.generate(), plain)


def test_speculation_drafts_never_touch_prefix(tiny_model):
    prompt = I.uniform_prompt(32, TINY.vocab, TINY.mask_id, seed=22)
    sched = O.OracleSched(steps_per_block=16, spec_blocks=2, spec_trigger=8, theta_remask=0.5, remask_max=1)
    sess = O.Session(tiny_model, sched, prompt, 128)
    sess.prefill()
    nblk, spec_steps, steps = 0, 0, 0
    while sess.begin_block():
        tok, st, kv = sess.state()
        assert kv == 32 + 32 * nblk
        c0 = 32 + 32 * nblk
        assert not (st[c0:c0 + 32] == O.DRAFT).any()  # accepted drafts became COMMITTED
        while True:
            out = sess.step()
            w = sess.window()
            steps += 1
            spec_steps += w["spec_on"]
            assert w["T"] in (32, 64, 96)
            assert sess.state()[2] == kv  # drafts never extend the prefix
            tok, st, _ = sess.state()
            assert not (st[:c0] == O.DRAFT).any()
            if out["block_done"]:
                break
        assert sess.window()["step"] <= 16
        nblk += 1
    assert nblk == 4 and spec_steps > 0
    tok, st, kv = sess.state()
    assert kv == 160 and not (tok[32:] == TINY.mask_id).any()


def test_revision_zero_threshold_equals_no_revision(tiny_model):
    prompt = I.uniform_prompt(32, TINY.vocab, TINY.mask_id, seed=23)
    a = O.Session(tiny_model, O.OracleSched(steps_per_block=8), prompt, 64).generate()
    b = O.Session(tiny_model, O.OracleSched(steps_per_block=8, theta_remask=0.0, theta_stable=0.0), prompt,
                  64).generate()
    assert np.array_equal(a, b)


# ------------------------------------------------------------ threshold commit (Sec. 3.3)
def _threshold(theta_visible=0.7, theta_stable=0.9, **kw):
    return O.OracleSched(commit_mode=1, theta_visible=theta_visible, theta_stable=theta_stable, **kw)


def test_threshold_commit_worked_case(oracle_lib):
    # a block of eight masked positions, the paper's default thresholds (0.7 visible, 0.9 stable)
    n, c0, c1 = 12, 2, 10
    st = np.full(n, O.MASKED, np.uint8)
    st[:c0] = O.FIXED
    st[c1:] = O.FIXED
    tok = np.where(st == O.MASKED, TINY.mask_id, 3).astype(np.int32)
    conf = np.array([0, 0, 0.95, 0.8, 0.6, 0.2, 0.9, 0.6999, 0.7, 0.5, 0, 0], np.float32)
    x0 = np.arange(100, 100 + n, dtype=np.int32)
    tok2, st2, out = O.commit(_threshold(), TINY.mask_id, tok, st, 0, n, c0, c1, 0, x0, conf, np.zeros(n, np.float32))
    want = [O.FIXED, O.FIXED, O.STABLE, O.COMMITTED, O.MASKED, O.MASKED, O.STABLE, O.MASKED, O.COMMITTED, O.MASKED,
            O.FIXED, O.FIXED]
    assert st2.tolist() == want
    assert tok2.tolist() == [3, 3, 102, 103, TINY.mask_id, TINY.mask_id, 106, TINY.mask_id, 108, TINY.mask_id, 3, 3]
    assert out["n_committed"] == 4 and out["n_stable"] == 2 and out["masked_after"] == 4 and not out["block_done"]


def test_threshold_fallback_promotes_the_most_confident(oracle_lib):
    # nothing reaches theta_visible: exactly one position, the first of the most confident, becomes visible
    n, c0, c1 = 10, 0, 10
    st = np.full(n, O.MASKED, np.uint8)
    tok = np.full(n, TINY.mask_id, np.int32)
    conf = np.array([0.1, 0.5, 0.3, 0.5, 0.2, 0.0, 0.5, 0.4, 0.1, 0.1], np.float32)
    x0 = np.arange(n, dtype=np.int32) + 7
    tok2, st2, out = O.commit(_threshold(), TINY.mask_id, tok, st, 0, n, c0, c1, 5, x0, conf, np.zeros(n, np.float32))
    assert out["n_committed"] == 1 and out["n_stable"] == 0 and out["masked_after"] == 9
    assert st2[1] == O.COMMITTED and tok2[1] == 8
    assert int((st2 == O.MASKED).sum()) == 9


@pytest.mark.parametrize("seed", range(6))
def test_threshold_reduces_to_the_schedule_rule(oracle_lib, seed):
    # theta_visible = 0: every masked position is taken, as the schedule does on a block's last step;
    # theta_visible unreachable: one per step, the schedule's top-1 (k = 1 when m steps are left)
    n, c0, c1 = 48, 8, 40
    rng = np.random.default_rng(seed)
    st = np.where(rng.random(n) < 0.6, O.MASKED, O.COMMITTED).astype(np.uint8)
    tok = np.where(st == O.MASKED, TINY.mask_id, 1).astype(np.int32)
    conf = I.scripted_confidences(n, seed=seed, ties=True)
    x0 = rng.integers(0, 1000, n).astype(np.int32)
    tc = np.zeros(n, np.float32)
    m = int((st[c0:c1] == O.MASKED).sum())
    S = 64
    all_t = O.commit(_threshold(0.0, 2.0, steps_per_block=S), TINY.mask_id, tok, st, 0, n, c0, c1, 0, x0, conf, tc)
    all_s = O.commit(O.OracleSched(steps_per_block=S), TINY.mask_id, tok, st, 0, n, c0, c1, S - 1, x0, conf, tc)
    assert np.array_equal(all_t[0], all_s[0]) and np.array_equal(all_t[1], all_s[1])
    assert all_t[2]["n_committed"] == m and all_t[2]["block_done"]
    one_t = O.commit(_threshold(2.0, 2.0, steps_per_block=S), TINY.mask_id, tok, st, 0, n, c0, c1, 0, x0, conf, tc)
    one_s = O.commit(O.OracleSched(steps_per_block=S), TINY.mask_id, tok, st, 0, n, c0, c1, S - m, x0, conf, tc)
    assert np.array_equal(one_t[0], one_s[0]) and np.array_equal(one_t[1], one_s[1])
    assert one_t[2]["n_committed"] == 1


def test_threshold_session_blocks_progress_and_finish(tiny_model):
    # unreachable visibility: one commit per step, block_len steps per block; theta_visible = 0: one step
    prompt = I.uniform_prompt(32, TINY.vocab, TINY.mask_id, seed=31)
    for tv, steps_per_block in ((2.0, 32), (0.0, 1)):
        sess = O.Session(tiny_model, _threshold(tv, 2.0, steps_per_block=8), prompt, 64)
        sess.prefill()
        blocks = 0
        while sess.begin_block():
            counts = []
            while True:
                out = sess.step()
                counts.append(out["n_committed"])
                assert out["n_committed"] >= 1
                if out["block_done"]:
                    break
            assert len(counts) == steps_per_block and sum(counts) == 32
            blocks += 1
        tok, st, kv = sess.state()
        assert blocks == 2 and kv == 96 and not (tok[32:] == TINY.mask_id).any()


# ------------------------------------------------------------ sparse cache refresh (Sec. 3.3)
def _scr_session(model, scr_rows, seed=51, **kw):
    prompt = I.uniform_prompt(32, TINY.vocab, TINY.mask_id, seed=seed)
    sess = O.Session(model, O.OracleSched(steps_per_block=4, scr_rows=scr_rows, **kw), prompt, 96)
    sess.prefill()
    assert sess.begin_block()
    while not sess.step()["block_done"]:
        pass
    assert sess.begin_block()  # the first block is prefix now: its tokens are visible, not stable
    return sess


def test_scr_merge_is_not_visible_within_the_step(tiny_model):
    # the tracked rows are queries only: the window's logits are those of a session without them
    a = _scr_session(tiny_model, 8, theta_stable=2.0)
    b = _scr_session(tiny_model, 0, theta_stable=2.0)
    ka, kb = a.prefix_kv(1, 0).copy(), b.prefix_kv(1, 0).copy()
    assert np.array_equal(ka, kb)
    k0 = a.prefix_kv(0, 0).copy()
    oa, ob = a.step(keep_logits=True), b.step(keep_logits=True)
    da, db = a.decisions(logits=True), b.decisions(logits=True)
    assert np.array_equal(da["logits"], db["logits"])
    assert {k: oa[k] for k in ("n_committed", "block_done", "masked_after")} == \
        {k: ob[k] for k in ("n_committed", "block_done", "masked_after")}
    assert oa["n_refreshed"] == 8 and ob["n_refreshed"] == 0
    # after the step the refreshed rows of layer 1 differ from the appended ones, the others do
    # not; layer 0's K/V depend on the token and its position only, so its refresh changes nothing
    ka2 = a.prefix_kv(1, 0)
    pos = a.scr_decisions()["pos"]
    changed = np.flatnonzero(np.abs(ka2 - ka).max(axis=1) > 0)
    assert set(changed.tolist()) == set(pos.tolist())
    assert np.array_equal(a.prefix_kv(0, 0), k0)


def test_scr_tracks_the_first_visible_prefix_positions(tiny_model):
    sess = _scr_session(tiny_model, 5, theta_stable=2.0)
    tok, st, kv = sess.state()
    sess.step()
    pos = sess.scr_decisions()["pos"]
    want = [p for p in range(kv) if st[p] == O.COMMITTED][:5]
    assert pos.tolist() == want and len(want) == 5


def test_scr_stable_threshold_zero_stabilizes_every_tracked_row(tiny_model):
    sess = _scr_session(tiny_model, 6, theta_stable=0.0)
    _, st0, kv = sess.state()
    visible = [p for p in range(kv) if st0[p] == O.COMMITTED]
    seen = []
    for _ in range(3):
        out = sess.step()
        pos = sess.scr_decisions()["pos"].tolist()
        assert out["n_refreshed"] == len(pos) and out["n_revised"] == 0
        seen += pos
        _, st, _ = sess.state()
        assert all(st[p] == O.STABLE for p in pos)
    assert seen == visible[:len(seen)] and len(seen) == min(18, len(visible))


def test_scr_revision_replaces_ids_and_skips_their_merge(tiny_model):
    # theta_remask above 1: every tracked row whose argmax differs from its id takes the argmax,
    # and only the rows that keep their id have their K/V merged
    sess = _scr_session(tiny_model, 8, theta_stable=2.0, theta_remask=1.5, remask_max=0)
    tok0, st0, _ = sess.state()
    k0 = sess.prefix_kv(1, 1).copy()
    out = sess.step()
    d = sess.scr_decisions()
    tok1, st1, _ = sess.state()
    k1 = sess.prefix_kv(1, 1)
    revised = [int(p) for p, x in zip(d["pos"], d["x0"]) if x != tok0[p]]
    kept = [int(p) for p, x in zip(d["pos"], d["x0"]) if x == tok0[p]]
    assert out["n_revised"] == len(revised) and out["n_refreshed"] == len(kept) and len(revised) > 0
    for p, x in zip(d["pos"], d["x0"]):
        assert tok1[p] == x and st1[p] == O.COMMITTED
    moved = set(np.flatnonzero(np.abs(k1 - k0).max(axis=1) > 0).tolist())
    assert moved == set(kept)


# ------------------------------------------------------------ adaptive lookahead (Sec. 3.2)
def _lookahead_windows(model, **kw):
    prompt = I.uniform_prompt(32, TINY.vocab, TINY.mask_id, seed=71)
    sess = O.Session(model, O.OracleSched(steps_per_block=8, spec_blocks=3, spec_trigger=4, **kw), prompt, 160)
    sess.prefill()
    windows = []
    while sess.begin_block():
        while True:
            out = sess.step()
            windows.append(sess.window()["T"])
            if out["block_done"]:
                break
    return windows, sess.state()[0]


def test_adaptive_lookahead_takes_the_blocks_within_the_allowance(tiny_model):
    lat = (1.0, 1.05, 1.1, 2.0)  # step latency with 1, 2, 3, 4 blocks of window
    w, _ = _lookahead_windows(tiny_model, spec_allowance=0.12, spec_lat=lat)
    assert set(w) <= {32, 64, 96} and 96 in w  # two future blocks at most: 1.1 <= 1.12 < 2.0
    w5, _ = _lookahead_windows(tiny_model, spec_allowance=0.06, spec_lat=lat)
    assert set(w5) <= {32, 64} and 64 in w5


def test_adaptive_lookahead_reduces_to_fixed_and_to_none(tiny_model):
    # an allowance no table entry exceeds: every spec block, the fixed form; 0 with a rising
    # table: none, the plain block-wise decoding
    lat = (1.0, 1.05, 1.1, 2.0)
    fixed_w, fixed_tok = _lookahead_windows(tiny_model)
    wide_w, wide_tok = _lookahead_windows(tiny_model, spec_allowance=10.0, spec_lat=lat)
    assert wide_w == fixed_w and np.array_equal(wide_tok, fixed_tok)
    none_w, none_tok = _lookahead_windows(tiny_model, spec_allowance=0.0, spec_lat=lat)
    assert set(none_w) == {32}
    prompt = I.uniform_prompt(32, TINY.vocab, TINY.mask_id, seed=71)
    plain = O.Session(tiny_model, O.OracleSched(steps_per_block=8), prompt, 160).generate()
    assert np.array_equal(none_tok[32:], plain)


def test_continuous_sliding_frontier_and_cache(tiny_model):
    """Continuous sliding (Sec. 3.2): a window of one block's length starting at the cache
    frontier; after a step, the leading run of positions that were visible at the forward and
    still are joins the cache with exactly the K/V that forward computed (all layers; at layer
    0 also those of the id alone at its position); the window then reaches into the next block
    and drafts there; positions left of the window are never revised; the block end appends
    only what has not slid."""
    Lp, bl = 32, 32
    prompt = I.uniform_prompt(Lp, TINY.vocab, TINY.mask_id, seed=61)
    sched = O.OracleSched(steps_per_block=8, slide=1)
    sess = O.Session(tiny_model, sched, prompt, 2 * bl)
    sess.prefill()
    assert sess.begin_block()
    sess.step()
    assert sess.window()["kv_len"] == Lp  # nothing was visible at the forward
    tok, st, kv = sess.state()
    assert kv == Lp
    # teacher forcing: the first 5 block positions visible (and the 6th masked)
    tok[Lp:Lp + bl] = TINY.mask_id
    st[Lp:Lp + bl] = O.MASKED
    tok[Lp:Lp + 5] = [3, 14, 15, 92, 65]
    st[Lp:Lp + 5] = O.COMMITTED
    sess.set_state(tok, st)
    L = TINY.n_layers
    pk = np.stack([sess.prefix_kv(l, 0) for l in range(L)])
    pv = np.stack([sess.prefix_kv(l, 1) for l in range(L)])
    win_tok, win_pos = tok[Lp:Lp + bl].copy(), np.arange(Lp, Lp + bl, dtype=np.int32)
    ref = O.forward(tiny_model, win_tok, win_pos, prefix_k=pk, prefix_v=pv, want_kv=True, logits=False)
    out = sess.step()
    w = sess.window()
    assert w["w0"] == Lp and w["T"] == bl and w["kv_len"] == Lp + 5
    for l in range(L):
        for which, r in ((0, ref["k"]), (1, ref["v"])):
            got = sess.prefix_kv(l, which)[Lp:Lp + 5]
            assert np.array_equal(got, r[l][:5])
    alone = O.forward(tiny_model, win_tok[:5], win_pos[:5], want_kv=True, logits=False, n_layers_run=1)
    assert np.allclose(sess.prefix_kv(0, 0)[Lp:Lp + 5], alone["k"][0], rtol=1e-6, atol=1e-7)
    assert out["n_drafts"] == 0  # the window still ended at the block end
    # the next window: one block's length from the frontier, 5 positions into the next block
    out = sess.step()
    w = sess.window()
    assert w["w0"] == Lp + 5 and w["T"] == bl
    assert out["n_drafts"] == 1
    tok2, st2, _ = sess.state()
    assert (st2[2 * Lp:2 * Lp + 5] == O.DRAFT).sum() == 1 and (st2[2 * Lp + 5:] != O.DRAFT).all()
    kept = sess.prefix_kv(1, 0)[Lp:Lp + 5].copy()
    # the commit pass with the window 5 positions into its block and every visible position a
    # revision candidate: those left of the window are untouched, one inside is re-masked
    n, c0, c1, w0 = 96, 32, 64, 37
    st_c = np.full(n, O.MASKED, np.uint8)
    st_c[c0:c0 + 8] = O.COMMITTED
    tok_c = np.where(st_c == O.MASKED, TINY.mask_id, 5).astype(np.int32)
    T = 32
    tc = np.linspace(0.01, 0.3, T).astype(np.float32)
    s_rev = O.OracleSched(steps_per_block=8, theta_remask=0.5, remask_max=32, slide=1)
    tok_r, st_r, out_r = O.commit(s_rev, TINY.mask_id, tok_c, st_c, w0, T, c0, c1, 0,
                                  np.arange(T, dtype=np.int32), np.full(T, 0.5, np.float32), tc)
    assert (st_r[c0:w0] == O.COMMITTED).all() and (tok_r[c0:w0] == 5).all()
    assert out_r["n_remasked"] == 3  # positions 37..39, the visible ones inside the window
    # finish the block in the first session: the append covers only [kv_len, c1)
    tok, st, kv = sess.state()
    m = np.flatnonzero(st[Lp:Lp + bl] == O.MASKED) + Lp
    tok[m], st[m] = 7, O.COMMITTED
    sess.set_state(tok, st)
    front = sess.state()[2]
    assert sess.begin_block()
    assert sess.state()[2] == Lp + bl
    assert np.array_equal(sess.prefix_kv(1, 0)[Lp:Lp + 5], kept)
    assert front >= Lp + 5
