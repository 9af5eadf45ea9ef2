"""Kernel-level parity on the GPU, through the C ABI (include/dllm_ops.h):
the tcgen05 GEMM, the split-KV attention and the fused LM head against
numpy/oracle definitions on the same seeded inputs, and the commit pass
bit-exact against the oracle's."""
import numpy as np
import pytest

import dllm_inputs as I
import oracle as O

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def dev():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    import paper_2606_13740_gb300 as pkg
    pkg.lib()
    return torch.device("cuda:0")


def _bf16(rng, shape, scale=1.0):
    return torch.from_numpy((rng.standard_normal(shape) * scale).astype(np.float32)).to(torch.bfloat16)


def _f64(t):
    return t.float().cpu().numpy().astype(np.float64)


# ------------------------------------------------------------------ GEMM
@pytest.mark.parametrize("M,N,K,grid", [
    (128, 32, 64, 1), (256, 32, 256, 0), (200, 40, 688, 1), (200, 40, 688, 3), (200, 40, 688, 7),
    (1024, 96, 1024, 0), (768, 300, 256, 5), (512, 16, 4096, 152), (384, 520, 320, 0),
])
def test_gemm_matches_numpy(dev, M, N, K, grid):
    from paper_2606_13740_gb300 import dllm_op_gemm
    rng = np.random.default_rng(M * 7 + N * 3 + K + grid)
    W = _bf16(rng, (M, K), 0.05)
    X = _bf16(rng, (N, K))
    D = dllm_op_gemm(W.to(dev), X.to(dev), M, N, K, grid=grid).cpu().numpy()
    ref = _f64(X) @ _f64(W).T
    scale = np.sqrt((_f64(X) ** 2).sum(1))[:, None] * np.sqrt((_f64(W) ** 2).sum(1))[None, :]
    assert np.all(np.abs(D - ref) <= 1e-5 * scale + 1e-6), np.abs(D - ref).max()


@pytest.mark.parametrize("M,N,K", [(12288, 32, 4096), (24576, 32, 4096), (4096, 32, 12288), (4096, 1024, 4096)])
def test_gemm_llada_shapes_sampled(dev, M, N, K):
    """Full LLaDA-8B projection shapes (QKV, gate/up, down; batch-16 tokens)."""
    from paper_2606_13740_gb300 import dllm_op_gemm
    rng = np.random.default_rng(M + N + K)
    W = _bf16(rng, (M, K), 0.02)
    X = _bf16(rng, (N, K))
    D = dllm_op_gemm(W.to(dev), X.to(dev), M, N, K).cpu().numpy()
    rows = rng.choice(M, size=min(M, 512), replace=False)
    cols = rng.choice(N, size=min(N, 48), replace=False)
    ref = _f64(X[cols]) @ _f64(W[rows]).T
    got = D[np.ix_(cols, rows)]
    assert np.abs(got - ref).max() <= 1e-4 * np.abs(ref).max()
    # deterministic: a second launch gives the same bits
    D2 = dllm_op_gemm(W.to(dev), X.to(dev), M, N, K).cpu().numpy()
    assert np.array_equal(D, D2)


def test_gemm_bounded_wait_times_out(dev):
    """A launch whose operand wait can never be satisfied (a flag nothing writes) gives up after
    its bounded wait, unwinds every role and reports DLLM_ETIMEOUT; the next launch is normal."""
    from paper_2606_13740_gb300.dllm import DllmError, dllm_op_gemm, dllm_op_gemm_timed
    M, N, K = 1024, 32, 1024
    rng = np.random.default_rng(5)
    W = _bf16(rng, (M, K), 0.05)
    X = _bf16(rng, (N, K))
    with pytest.raises(DllmError) as e:
        dllm_op_gemm_timed(W.to(dev), X.to(dev), M, N, K, 1, flags=4)
    assert e.value.code == -4
    D = dllm_op_gemm(W.to(dev), X.to(dev), M, N, K).cpu().numpy()
    ref = _f64(X) @ _f64(W).T
    scale = np.sqrt((_f64(X) ** 2).sum(1))[:, None] * np.sqrt((_f64(W) ** 2).sum(1))[None, :]
    assert np.all(np.abs(D - ref) <= 1e-5 * scale + 1e-6)


# ------------------------------------------------------------------ attention
def _attn_ref(q, k, v, kv_len, T):
    B, H, _, hd = q.shape
    out = np.zeros((B * T, H * hd))
    for b in range(B):
        nk = kv_len[b] + T
        for h in range(H):
            s = q[b, h] @ k[b, h, :nk].T / np.sqrt(hd)
            s -= s.max(1, keepdims=True)
            p = np.exp(s)
            p /= p.sum(1, keepdims=True)
            out[b * T:(b + 1) * T, h * hd:(h + 1) * hd] = p @ v[b, h, :nk]
    return out


@pytest.mark.parametrize("B,T,H,hd,kv,cap", [
    (1, 32, 4, 128, [512], 600), (2, 96, 2, 64, [0, 37], 160), (1, 512, 2, 128, [0], 512),
    (3, 32, 2, 128, [5, 300, 1000], 1100), (2, 64, 4, 128, [4096, 4096], 4160), (1, 1, 1, 64, [3], 8),
    # the tensor-core kernel (head dim 128, >= 1024 keys): two 128-row query tiles (the second
    # ragged), eight key splits per cluster, a sequence whose keys fill no split but the first
    (1, 192, 2, 128, [1100], 1300), (1, 32, 1, 128, [2000], 2048), (2, 40, 3, 128, [1, 1500], 1600),
    # more units than one wave (12 x 32 = 384 > 2 per SM), mixed prefix lengths
    (12, 64, 32, 128, [1000, 1200, 2000, 964, 1100, 1500, 1960, 1024, 1300, 999, 1700, 1800], 2100),
])
def test_attention_matches_numpy(dev, B, T, H, hd, kv, cap):
    from paper_2606_13740_gb300 import dllm_op_attention
    rng = np.random.default_rng(B * 100 + T + hd)
    q = _bf16(rng, (B, H, T, hd))
    k = _bf16(rng, (B, H, cap, hd))
    v = _bf16(rng, (B, H, cap, hd))
    kv_len = torch.tensor(kv, dtype=torch.int32)
    out = dllm_op_attention(q.to(dev), k.to(dev), v.to(dev), kv_len.to(dev), B, T, H, hd, cap, max(kv))
    got = out.float().cpu().numpy()
    ref = _attn_ref(_f64(q), _f64(k), _f64(v), kv, T)
    rel = np.linalg.norm(got - ref) / np.linalg.norm(ref)
    assert rel <= 1e-2, rel
    assert np.abs(got - ref).max() <= 0.05 * np.abs(ref).max()


# ------------------------------------------------------------------ LM head
@pytest.mark.parametrize("V,N,d,mask", [(1024, 32, 256, 1023), (126464, 32, 4096, 126463), (2048, 96, 512, 0)])
def test_lmhead_decision_matches_oracle(dev, V, N, d, mask):
    from paper_2606_13740_gb300 import dllm_op_lmhead
    rng = np.random.default_rng(V + N)
    W = _bf16(rng, (V, d), 0.02)
    X = _bf16(rng, (N, d))
    cur = rng.integers(0, V, N).astype(np.int32)
    cur[::5] = mask
    x0, conf, tc, lg = dllm_op_lmhead(W.to(dev), X.to(dev), torch.from_numpy(cur).to(dev), V, N, d, mask,
                                      want_logits=(V <= 2048))
    x0, conf, tc = x0.cpu().numpy(), conf.cpu().numpy(), tc.cpu().numpy()
    ref_logits = (_f64(X) @ _f64(W).T).astype(np.float32)
    if lg is not None:
        assert np.abs(lg.cpu().numpy() - ref_logits).max() <= 1e-4 * np.abs(ref_logits).max()
    for n in range(N):
        rx0, rconf, rtc, margin = O.decide(ref_logits[n], mask, cur[n])
        assert x0[n] != mask
        if margin > 1e-3:
            assert x0[n] == rx0
        assert abs(conf[n] - rconf) <= 1e-3 * rconf
        assert abs(tc[n] - rtc) <= 1e-3 * max(rtc, 1e-30) + 1e-12


# ------------------------------------------------------------------ commit
def _random_case(rng, use_cache, spec_blocks):
    bl = 32
    if use_cache:
        c0 = 64 + bl * int(rng.integers(0, 3))
        w0 = c0
        nspec = spec_blocks if spec_blocks else 0
        T = bl * (1 + nspec)
        n_pos = w0 + T + int(rng.integers(0, 40))
    else:
        w0, c0 = 0, 16 + bl * int(rng.integers(0, 2))
        n_pos = c0 + bl * 2
        T = n_pos
    c1 = c0 + bl
    st = rng.choice(np.array([1, 1, 1, 2, 2, 3, 4], np.uint8), size=n_pos)
    st[:min(c0, 16)] = 0
    tok = np.where(st == 1, 1023, rng.integers(0, 1000, n_pos)).astype(np.int32)
    x0 = rng.integers(0, 1023, T).astype(np.int32)
    conf = I.scripted_confidences(T, int(rng.integers(1 << 30)), ties=bool(rng.integers(0, 2)))
    tokconf = I.scripted_confidences(T, int(rng.integers(1 << 30)), ties=True)
    return tok, st, w0, T, c0, c1, x0, conf, tokconf


@pytest.mark.parametrize("seed", range(40))
def test_commit_bit_exact_vs_oracle(dev, seed):
    from paper_2606_13740_gb300 import Sched, dllm_op_commit
    rng = np.random.default_rng(seed)
    use_cache = int(seed % 4 != 3)
    spec = int(rng.integers(0, 3)) if use_cache else 0
    S = int(rng.choice([4, 8, 32]))
    step = int(rng.integers(0, S))
    theta = float(rng.choice([0.0, 0.5]))
    rmax = int(rng.integers(1, 4))
    tok, st, w0, T, c0, c1, x0, conf, tokconf = _random_case(rng, use_cache, spec)
    gs = Sched(steps_per_block=S, theta_remask=theta, theta_stable=0.9, remask_max=rmax, spec_blocks=spec,
               use_prefix_cache=use_cache)
    os_ = O.OracleSched(steps_per_block=S, block_len=32, theta_remask=theta, theta_stable=0.9, remask_max=rmax,
                        spec_blocks=spec, use_prefix_cache=use_cache)
    gt, gst, gout = dllm_op_commit(gs, 1023, tok, st, w0, T, c0, c1, step, x0, conf, tokconf)
    ot, ost, oout = O.commit(os_, 1023, tok, st, w0, T, c0, c1, step, x0, conf, tokconf)
    assert np.array_equal(gst, ost)
    assert np.array_equal(gt, ot)
    assert gout == {k: oout[k] for k in gout}


@pytest.mark.parametrize("seed", range(40))
def test_commit_threshold_bit_exact_vs_oracle(dev, seed):
    """Staged token stabilization (Sec. 3.3) on random states, ties included: the same
    positions become visible / stable, the same fallback position, the same counts."""
    from paper_2606_13740_gb300 import COMMIT_THRESHOLD, Sched, dllm_op_commit
    rng = np.random.default_rng(1000 + seed)
    use_cache = int(seed % 4 != 3)
    spec = int(rng.integers(0, 3)) if use_cache else 0
    S = int(rng.choice([4, 8, 32]))
    step = int(rng.integers(0, S))
    theta = float(rng.choice([0.0, 0.5]))
    rmax = int(rng.integers(1, 4))
    tv = float(rng.choice([0.0, 0.3, 0.5, 0.75, 2.0]))
    ts = float(rng.choice([0.5, 0.9, 2.0]))
    tok, st, w0, T, c0, c1, x0, conf, tokconf = _random_case(rng, use_cache, spec)
    gs = Sched(steps_per_block=S, theta_remask=theta, theta_stable=ts, remask_max=rmax, spec_blocks=spec,
               use_prefix_cache=use_cache, commit_mode=COMMIT_THRESHOLD, theta_visible=tv)
    os_ = O.OracleSched(steps_per_block=S, block_len=32, theta_remask=theta, theta_stable=ts, remask_max=rmax,
                        spec_blocks=spec, use_prefix_cache=use_cache, commit_mode=1, theta_visible=tv)
    gt, gst, gout = dllm_op_commit(gs, 1023, tok, st, w0, T, c0, c1, step, x0, conf, tokconf)
    ot, ost, oout = O.commit(os_, 1023, tok, st, w0, T, c0, c1, step, x0, conf, tokconf)
    assert np.array_equal(gst, ost)
    assert np.array_equal(gt, ot)
    assert gout == {k: oout[k] for k in gout}
    m = int((st[c0:c1] == 1).sum())
    if m:
        assert gout["n_committed"] >= 1  # every step makes progress
