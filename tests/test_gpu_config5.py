"""Batch-16 step with a long synthetic prefix (the wide-tile, tensor-bound path), on the GPU
through the C ABI, at full LLaDA-8B width with two layers:

- 16 sequences, each with 4096 cached prefix positions of synthetic K/V (seeded generator,
  identical on both sides), a 64-token window (current block + one speculative block) with
  32 masked positions and Zipf(1.1) ids elsewhere;
- one denoising step: window and commit counts exact; for two sampled sequences the oracle
  runs the same forward (same tokens, positions and prefix) and the logits agree within 1e-2
  relative L2, argmax equal wherever the oracle's top-1/top-2 margin exceeds 0.05;
- every sequence's step is independent of the others: changing the other fifteen
  sequences' window ids leaves sequence 0's logits bit-identical.
"""
import numpy as np
import pytest

import dllm_inputs as I
import oracle as O

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

SHAPE = dict(d_model=4096, n_heads=32, head_dim=128, ffn=12288, vocab=126464, mask_id=126463, rope_base=500000.0)
B, P, T, L = 16, 4096, 64, 2


@pytest.fixture(scope="module")
def gpu():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    import paper_2606_13740_gb300 as pkg
    pkg.lib()
    return pkg


def _window_state(cfg, tok, st, seqs, id_seed=I.SEED_ZIPF, visible=O.COMMITTED):
    win = np.arange(P, P + T)
    ids = I.zipf_ids((B, T), cfg.vocab, cfg.mask_id, seed=id_seed)
    ids[0] = I.zipf_ids((B, T), cfg.vocab, cfg.mask_id)[0]  # sequence 0 keeps its ids
    for k, b in enumerate(seqs):
        tok[k, win] = ids[b]
        st[k, win] = visible
        m = win[I.masked_positions(T, 32, seed=I.SEED_PROMPT + 100 + b)]
        tok[k, m], st[k, m] = cfg.mask_id, O.MASKED
    return tok, st


def _step(gpu, seqs, id_seed=I.SEED_ZIPF, visible=O.COMMITTED, sls=0):
    cfg = gpu.Config(n_layers=L, max_batch=len(seqs), max_ctx=P + T, max_window=T, **SHAPE)
    ctx = gpu.Context(cfg)
    sched = gpu.Sched(steps_per_block=32, spec_trigger=32, spec_blocks=1, sls=sls)
    ctx.dllm_set_prefix_kv_random(sched, len(seqs), P, T, I.SEED_KV)
    ctx.dllm_begin_block()
    tok, st, _ = ctx.dllm_get_state()
    tok, st = _window_state(cfg, tok, st, seqs, id_seed, visible)
    ctx.dllm_set_state(tok, st)
    ctx.dllm_set_debug(0 if sls else 1)  # captured logits would switch the skipping off
    out = ctx.dllm_denoise_step()
    w = ctx.dllm_window()
    d = ctx.dllm_get_step_debug(logits=not sls)
    ctx.close()
    return tok, st, out, w, d


def _oracle_prefix(b, layer, which):
    # the GPU's synthetic prefix: tensor 2^32 + (b*L + layer)*2 + which, element pos*qd + h*hd + i
    tid = (1 << 32) + (b * L + layer) * 2 + which
    bits = O.gen_bf16(I.SEED_KV, tid, 0, P * 4096, 1.0)
    return O.bf16_to_f32(bits).reshape(P, 4096)


def test_batch16_long_prefix_step_matches_oracle(gpu):
    seqs = list(range(B))
    tok, st, out, w, d = _step(gpu, seqs)
    assert w["T"] == T and w["w0"] == P and w["spec_on"] == 1 and w["kv_len"] == P
    # k = ceil(m / S) commits per sequence at step 0 (m masked in the current block, S = 32)
    assert out["n_committed"] == sum(-(-int((st[b, P:P + 32] == O.MASKED).sum()) // 32) for b in seqs)
    assert not (d["x0"] == SHAPE["mask_id"]).any()
    model = O.Model(O.OracleConfig(n_layers=L, **SHAPE))
    for b in (0, 13):
        pk = np.stack([_oracle_prefix(b, l, 0) for l in range(L)])
        pv = np.stack([_oracle_prefix(b, l, 1) for l in range(L)])
        ref = O.forward(model, tok[b, P:P + T], np.arange(P, P + T), prefix_k=pk, prefix_v=pv)["logits"]
        got = d["logits"][b]
        rel = float(np.linalg.norm(got - ref) / np.linalg.norm(ref))
        assert rel <= 1e-2, (b, rel)
        dec = [O.decide(ref[t], SHAPE["mask_id"], int(tok[b, P + t])) for t in range(T)]
        x0 = np.array([v[0] for v in dec])
        safe = np.array([v[3] for v in dec]) > 0.05
        assert safe.sum() > 0
        assert np.array_equal(d["x0"][b][safe], x0[safe]), b


def test_batch16_sequences_independent(gpu):
    _, _, _, _, da = _step(gpu, list(range(B)))
    _, _, _, _, db = _step(gpu, list(range(B)), id_seed=I.SEED_ZIPF + 17)
    assert not np.array_equal(da["x0"][1:], db["x0"][1:])  # the others did change
    assert np.array_equal(da["logits"][0], db["logits"][0])
    assert np.array_equal(da["x0"][0], db["x0"][0]) and np.array_equal(da["conf"][0], db["conf"][0])


def test_batch16_selective_logits_skipping_matches_oracle(gpu):
    """The same full-width batch-16 step with the visible half of every window STABLE and
    selective logits skipping on: the head runs over the 512 masked rows only; those rows'
    decisions match the oracle's for the sampled sequences, the STABLE rows carry none."""
    seqs = list(range(B))
    tok, st, out, w, d = _step(gpu, seqs, visible=O.STABLE, sls=1)
    model = O.Model(O.OracleConfig(n_layers=L, **SHAPE))
    for b in (0, 13):
        need = st[b, P:P + T] == O.MASKED
        assert need.sum() == 32
        assert (d["x0"][b][~need] == -1).all() and (d["conf"][b][~need] == 0).all()
        pk = np.stack([_oracle_prefix(b, l, 0) for l in range(L)])
        pv = np.stack([_oracle_prefix(b, l, 1) for l in range(L)])
        ref = O.forward(model, tok[b, P:P + T], np.arange(P, P + T), prefix_k=pk, prefix_v=pv)["logits"]
        dec = [O.decide(ref[t], SHAPE["mask_id"], int(tok[b, P + t])) for t in range(T)]
        x0 = np.array([v[0] for v in dec])
        conf = np.array([v[1] for v in dec])
        safe = need & (np.array([v[3] for v in dec]) > 0.05)
        assert safe.sum() > 0
        assert np.array_equal(d["x0"][b][safe], x0[safe]), b
        assert np.allclose(d["conf"][b][need], conf[need], rtol=0.05), b
