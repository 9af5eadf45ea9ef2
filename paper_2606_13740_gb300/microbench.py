"""Single-kernel micro-benchmarks through the C ABI (dllm_ops.h).

    python -m paper_2606_13740_gb300.microbench gemm --M 24576 --N 32 --K 4096 --reps 3

Draws seeded bf16 operands on the device and runs the entry point `reps`
times; prints the wall time per call (which includes the op's own scratch
allocation and synchronisation: use ncu or the profiled step for kernel time).
"""
from __future__ import annotations

import argparse
import json
import time

import torch

from .dllm import dllm_op_attention, dllm_op_gemm, dllm_op_gemm_timed, dllm_op_gemm_trace, lib


def main(argv=None):
    ap = argparse.ArgumentParser()
    ap.add_argument("op", choices=("gemm", "attention", "gemm-sweep", "gemm-trace", "step-trace", "step-small",
                                   "step-b16", "window-sweep", "generate"))
    ap.add_argument("--layers", type=int, default=32)
    ap.add_argument("--M", type=int, default=24576)
    ap.add_argument("--N", type=int, default=32)
    ap.add_argument("--K", type=int, default=4096)
    ap.add_argument("--B", type=int, default=16)
    ap.add_argument("--T", type=int, default=64, help="attention / step-trace: window tokens")
    ap.add_argument("--H", type=int, default=32)
    ap.add_argument("--P", type=int, default=4096)
    ap.add_argument("--reps", type=int, default=3)
    ap.add_argument("--dump", default="", help="gemm-trace: write every CTA's timeline to this JSON file")
    ap.add_argument("--no-pdl", action="store_true")
    ap.add_argument("--debug", type=int, default=0, help="step-trace: extra dllm_set_debug flags")
    ap.add_argument("--lat", type=float, nargs="*", default=[3.37, 3.97, 4.14],
                    help="generate: step ms with a window of 1, 2, 3 blocks (the window sweep at batch 1)")
    ap.add_argument("--allowance", type=float, default=0.2, help="generate: adaptive lookahead allowance")
    ap.add_argument("--sls", type=int, default=0, help="step-b16: selective logits skipping (0/1)")
    ap.add_argument("--stable", action="store_true", help="step-b16: the window's visible positions are STABLE")
    a = ap.parse_args(argv)
    lib()
    dev = torch.device("cuda:0")
    g = torch.Generator(device=dev)
    g.manual_seed(0)
    if a.op == "gemm-sweep":
        # kernel time vs weight rows: separates the fixed cost of a launch from the streaming rate;
        # flags: 0 plain launches (113 KB), 1 PDL chain (113 KB), 2 plain (227 KB), 3 PDL chain (227 KB)
        rows = []
        for K in (4096, 12288):
            for M in (1024, 4096, 12288, 24576, 126464):
                if M * K > 126464 * 4096:
                    continue
                W = (torch.randn(M, K, device=dev, generator=g) * 0.02).to(torch.bfloat16)
                X = torch.randn(a.N, K, device=dev, generator=g).to(torch.bfloat16)
                r = {"M": M, "N": a.N, "K": K}
                for flags in (0, 1, 2, 3):
                    ms, _ = dllm_op_gemm_timed(W, X, M, a.N, K, a.reps, flags=flags)
                    r[f"us_f{flags}"] = round(ms * 1e3, 2)
                r["GBps_best"] = round(M * K * 2 / (min(r[f"us_f{f}"] for f in range(4)) * 1e-6) / 1e9)
                rows.append(r)
                del W, X
        print(json.dumps({"op": "gemm-sweep", "rows": rows}))
        return
    if a.op == "step-small":
        step_small(a)
        return
    if a.op == "step-b16":
        step_b16(a)
        return
    if a.op == "window-sweep":
        window_sweep(a)
        return
    if a.op == "generate":
        generate(a)
        return
    if a.op == "step-trace":
        step_trace(a)
        return
    if a.op == "gemm-trace":
        # per-CTA timeline of one launch (microseconds from the first CTA's entry)
        W = (torch.randn(a.M, a.K, device=dev, generator=g) * 0.02).to(torch.bfloat16)
        X = torch.randn(a.N, a.K, device=dev, generator=g).to(torch.bfloat16)
        ms, tr = dllm_op_gemm_trace(W, X, a.M, a.N, a.K, a.reps)
        t0 = int(tr[:, 0].min())
        if a.dump:
            rows = []
            for r in tr.astype("int64"):
                rel = [round((x - t0) / 1e3, 3) if x > 0 else None for x in r[[0, 1, 2, 3, 4, 5, 7, 8, 9, 10, 11]]]
                rows.append({"sm": int(r[6]), "last": int(r[12]), "tile": int(r[13]), "t": rel})
            with open(a.dump, "w") as f:
                json.dump({"cols": ["start", "prologue", "first_data", "last_data", "epi_done", "exit", "dep_wait",
                                    "acc_ready", "part_stored", "ticket", "reduced"], "ctas": rows}, f)
        names = ("start", "prologue", "first_data", "last_data", "epi_done", "exit")
        rel = {n: ((tr[:, i].astype("int64") - t0) / 1e3) for i, n in enumerate(names)}
        rel["dep_wait"] = (tr[:, 7].astype("int64") - t0) / 1e3
        summary = {n: {"min": float(v.min()), "median": float(sorted(v)[len(v) // 2]), "max": float(v.max())}
                   for n, v in rel.items()}
        print(json.dumps({"op": "gemm-trace", "M": a.M, "N": a.N, "K": a.K, "us_per_launch": ms * 1e3,
                          "ctas": int(len(tr)), "sms": sorted(set(int(x) for x in tr[:, 6]))[:4],
                          "timeline_us": summary}))
        return
    if a.op == "gemm":
        W = (torch.randn(a.M, a.K, device=dev, generator=g) * 0.02).to(torch.bfloat16)
        X = torch.randn(a.N, a.K, device=dev, generator=g).to(torch.bfloat16)
        call = lambda: dllm_op_gemm(W, X, a.M, a.N, a.K)  # noqa: E731
        nbytes = a.M * a.K * 2
    else:
        hd, cap = 128, a.P + a.T
        q = torch.randn(a.B, a.H, a.T, hd, device=dev, generator=g).to(torch.bfloat16)
        k = torch.randn(a.B, a.H, cap, hd, device=dev, generator=g).to(torch.bfloat16)
        v = torch.randn(a.B, a.H, cap, hd, device=dev, generator=g).to(torch.bfloat16)
        kv = torch.full((a.B,), a.P, dtype=torch.int32, device=dev)
        call = lambda: dllm_op_attention(q, k, v, kv, a.B, a.T, a.H, hd, cap, a.P)  # noqa: E731
        nbytes = 2 * a.B * a.H * cap * hd * 2
    torch.cuda.synchronize()
    times = []
    for _ in range(a.reps):
        t0 = time.perf_counter()
        call()
        torch.cuda.synchronize()
        times.append(time.perf_counter() - t0)
    print(json.dumps({"op": a.op, "wall_ms_per_call": [t * 1e3 for t in times], "bytes": nbytes}))



SHAPE_8B = dict(d_model=4096, n_heads=32, head_dim=128, ffn=12288, vocab=126464, mask_id=126463, rope_base=500000.0)


def _timed_steps(ctx, step, n, warm=3):
    import torch
    for _ in range(warm):
        step()
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(ctx.stream)
    for _ in range(n):
        step()
    e1.record(ctx.stream)
    torch.cuda.synchronize()
    return e0.elapsed_time(e1) / n


def step_b16(a):
    """Batch-16 denoising step: synthetic prefix KV of 4096 positions per sequence, a 64-token
    window (current block + one speculative block) with 32 masked, Zipf(1.1) ids; the other 32
    visible (COMMITTED, or STABLE with --stable).  Prints ms/step and the projections' achieved
    bf16 TFLOP/s (events around each launch; the LM head counted over the rows it decides)."""
    import numpy as np

    import dllm_inputs as I

    from .dllm import COMMITTED, MASKED, STABLE, Config, Context, Sched

    B, P, T, L = 16, 4096, 64, a.layers
    cfg = Config(max_batch=B, max_ctx=P + T, max_window=T, n_layers=L, **SHAPE_8B)
    ctx = Context(cfg)
    sched = Sched(steps_per_block=32, spec_trigger=32, spec_blocks=1, sls=a.sls)
    ctx.dllm_set_prefix_kv_random(sched, B, P, T, I.SEED_KV)
    ctx.dllm_begin_block()
    tok, st, _ = ctx.dllm_get_state()
    win = np.arange(P, P + T)
    tok[:, win] = I.zipf_ids((B, T), cfg.vocab, cfg.mask_id)
    st[:, win] = STABLE if a.stable else COMMITTED
    for b in range(B):
        m = win[I.masked_positions(T, 32, seed=I.SEED_PROMPT + 100 + b)]
        tok[b, m], st[b, m] = cfg.mask_id, MASKED
    ctx.dllm_set_state(tok, st)
    w = ctx.dllm_window()
    head_rows = B * T if not (a.sls and a.stable) else int((st[:, win] != STABLE).sum())

    def step():
        ctx.dllm_rewind_block()
        ctx.dllm_denoise_step(want_out=False)

    ms = _timed_steps(ctx, step, a.reps)
    ctx.dllm_set_profile(1)
    for _ in range(8):
        step()
    prof, psteps = ctx.dllm_get_profile()
    ctx.dllm_set_profile(0)
    N = B * T
    d, F, V = cfg.d_model, cfg.ffn, cfg.vocab
    layer_flops = 2 * N * (4 * d * d + 3 * d * F)
    head_flops = 2 * head_rows * V * d
    attn_flops = B * L * 4 * T * (P + T) * d
    chain_ms = (prof["qkv"]["ms_total"] + prof["layer"]["ms_total"] + prof["head"]["ms_total"]) / psteps
    gemm_flops = L * layer_flops + head_flops
    print(json.dumps({"op": "step-b16", "sls": a.sls, "stable": a.stable, "head_rows": head_rows,
                      "window": w, "ms_per_step": ms, "steps_per_s": 1e3 / ms,
                      "kernel_ms_per_step": {k: v["ms_total"] / psteps for k, v in prof.items()},
                      "gemm_tflops": gemm_flops / (chain_ms * 1e-3) / 1e12,
                      "attn_kv_GBps": B * L * 2 * (P + T) * d * 2 / (prof["attn"]["ms_total"] / psteps * 1e-3) / 1e9,
                      "step_tflops": (gemm_flops + L * 0 + attn_flops) / (ms * 1e-3) / 1e12}))
    ctx.close()


def window_sweep(a):
    """LLaDA-8B step time against the window length (512-token prefix, batch 1): flat while the
    projections stream weights, rising once the token tile makes them tensor-bound."""
    import numpy as np

    from .dllm import COMMITTED, MASKED, Config, Context, Sched

    rows = []
    for T in (32, 64, 96, 128, 192, 256):
        cfg = Config(max_batch=1, max_ctx=512 + T, max_window=max(T, 512), block_len=T, n_layers=a.layers,
                     **SHAPE_8B)
        ctx = Context(cfg)
        rng = np.random.default_rng(1)
        ctx.dllm_prefill(Sched(steps_per_block=T), rng.integers(0, 126463, 512).astype(np.int32), T)
        # one block of length T: the window is the whole block, every position masked
        ctx.dllm_begin_block()
        ctx.dllm_set_state(*ctx.dllm_get_state()[:2])  # rewind point
        w = ctx.dllm_window()

        def step():
            ctx.dllm_rewind_block()
            ctx.dllm_denoise_step(want_out=False)

        ms = _timed_steps(ctx, step, a.reps)
        rows.append({"T": T, "window": w["T"], "ms_per_step": round(ms, 4)})
        ctx.close()
    print(json.dumps({"op": "window-sweep", "rows": rows}))


def generate(a):
    """Whole generations through dllm_generate at LLaDA-8B shape: 256-token prompt, 4 blocks of
    32 with 32 steps per block (one commit per step); a 1024-token prompt, 8 blocks, with
    speculation (window 96 when <= 8 masked) and revision (theta 0.5, at most 1 per step); and
    the threshold commit rule (staged token stabilization) on the 256-token prompt with the
    paper's thresholds (0.7 visible, 0.9 stable; a random-weight model's confidences stay near
    1/V, so every step takes the single-position fallback) and with theta_visible 0 (a whole
    block per step: the rule's fastest case); and sparse cache refresh of 32 visible prefix
    positions per step (random weights never reach theta_stable, so from the second block on
    every step carries 32 refresh rows besides its 32-token window); and the 1024-token workload
    with adaptive lookahead from the window sweep's step times (--lat, --allowance)."""
    import time

    import numpy as np

    import dllm_inputs as I

    from .dllm import COMMIT_THRESHOLD, Config, Context, Sched

    out = []
    for name, Lp, gen, sched in (
            ("blocks_p256_g128", 256, 128, Sched(steps_per_block=32)),
            ("spec_revision_p1024_g256", 1024, 256,
             Sched(steps_per_block=32, spec_trigger=8, spec_blocks=2, theta_remask=0.5, remask_max=1)),
            ("threshold_0.7_0.9_p256_g128", 256, 128,
             Sched(steps_per_block=32, commit_mode=COMMIT_THRESHOLD, theta_visible=0.7, theta_stable=0.9)),
            ("threshold_0_p256_g128", 256, 128,
             Sched(steps_per_block=32, commit_mode=COMMIT_THRESHOLD, theta_visible=0.0, theta_stable=0.9)),
            ("scr32_p256_g128", 256, 128, Sched(steps_per_block=32, scr_rows=32)),
            ("slide_p256_g128", 256, 128, Sched(steps_per_block=32, slide=1)),
            ("slide_lookahead_p1024_g256", 1024, 256,
             Sched(steps_per_block=32, slide=1, spec_trigger=8, spec_blocks=2, theta_remask=0.5, remask_max=1)),
            ("adaptive_lookahead_p1024_g256", 1024, 256,
             Sched(steps_per_block=32, spec_trigger=8, spec_blocks=2, theta_remask=0.5, remask_max=1,
                   spec_allowance=a.allowance, spec_lat=tuple(a.lat)))):
        cfg = Config(max_batch=1, max_ctx=Lp + gen, max_window=max(Lp, 96 + sched.scr_rows), n_layers=a.layers,
                     **SHAPE_8B)
        ctx = Context(cfg)
        prompt = I.uniform_prompt(Lp, cfg.vocab, cfg.mask_id)
        ctx.dllm_generate(sched, prompt, gen)  # warm-up: graphs for every window shape
        ctx.dllm_sync()
        t0 = time.perf_counter()
        toks, stats = ctx.dllm_generate(sched, prompt, gen)
        dt = time.perf_counter() - t0
        out.append({"workload": name, "seconds": round(dt, 4), "gen_tokens_per_s": gen / dt,
                    "steps_per_s": stats["steps"] / dt, **stats})
        ctx.close()
    print(json.dumps({"op": "generate", "runs": out}))


def step_small(a):
    """A few denoising steps of a 2-layer model at the LLaDA-8B width (about 3 GB on the device):
    the small case for ncu captures of the step's kernels."""
    import numpy as np

    from .dllm import Config, Context, Sched

    shape = dict(n_layers=2, d_model=4096, n_heads=32, head_dim=128, ffn=12288, vocab=126464, mask_id=126463,
                 rope_base=500000.0)
    ctx = Context(Config(max_batch=1, max_ctx=544, max_window=512, **shape))
    rng = np.random.default_rng(1)
    ctx.dllm_prefill(Sched(steps_per_block=24), rng.integers(0, 126463, 512).astype(np.int32), 32)
    ctx.dllm_begin_block()
    for _ in range(a.reps):
        ctx.dllm_denoise_step(want_out=False)
    ctx.dllm_sync()
    ctx.close()
    print(json.dumps({"op": "step-small", "steps": a.reps}))


def step_trace(a):
    """Timeline of the GEMM launches inside one LLaDA-8B-shaped denoising step (B=1, 512-token
    prefix, 32-token window), relative to the step's first GEMM start (microseconds)."""
    import numpy as np

    from .dllm import COMMITTED, MASKED, Config, Context, Sched

    shape = dict(n_layers=32, d_model=4096, n_heads=32, head_dim=128, ffn=12288, vocab=126464, mask_id=126463,
                 rope_base=500000.0)
    T = a.T if a.T in (32, 64, 96, 128, 192, 256) else 32
    cfg = Config(max_batch=1, max_ctx=512 + T, max_window=512, block_len=T, **shape)
    ctx = Context(cfg)
    flags = 16 | (4 if a.no_pdl else 0) | a.debug
    ctx.dllm_set_debug(flags)
    rng = np.random.default_rng(1)
    prompt = rng.integers(0, cfg.vocab - 1, 512).astype(np.int32)
    ctx.dllm_prefill(Sched(steps_per_block=24), prompt, T)
    ctx.dllm_begin_block()
    for _ in range(4):
        ctx.dllm_denoise_step(want_out=False)
    ctx.dllm_sync()
    tr = ctx.dllm_get_trace().astype(np.int64)
    if a.dump:
        np.save(a.dump, tr)
    names = ["qkv", "attn", "oproj", "gateup", "down"] * 32 + ["head"]
    t0 = min(int(x[:, 0][x[:, 0] > 0].min()) for x in tr)
    rows = []
    prev_exit = None
    for i, x in enumerate(tr):
        v = x[x[:, 0] > 0]
        if i < len(names) and names[i] == "attn":  # slots: start, dep wait, loop end, ticket, merged
            rel = lambda c: (v[:, c][v[:, c] > 0] - t0) / 1e3  # noqa: E731
            r = {"k": "attn", "start_min": float(rel(0).min()), "depwait_med": float(np.median(rel(1))),
                 "loop_max": float(rel(2).max()), "ticket_max": float(rel(3).max()),
                 "merged_max": float(rel(4).max()) if (v[:, 4] > 0).any() else None}
            if prev_exit is not None:
                r["gap_prev_exit_to_depwait"] = r["depwait_med"] - prev_exit
            prev_exit = r["merged_max"] if r["merged_max"] is not None else r["loop_max"]
            rows.append({k: (round(v, 2) if isinstance(v, float) else v) for k, v in r.items()})
            continue
        rel = lambda c: (v[:, c][v[:, c] > 0] - t0) / 1e3  # noqa: E731
        r = {"k": names[i] if i < len(names) else str(i), "start_min": float(rel(0).min()),
             "start_max": float(rel(0).max()), "depwait_med": float(np.median(rel(7))),
             "first_data_med": float(np.median(rel(2))), "last_data_max": float(rel(3).max()),
             "epi_done_max": float(rel(4).max()),
             "exit_max": float(rel(5).max()) if (v[:, 5] > 0).any() else float(rel(4).max())}
        if prev_exit is not None:
            r["gap_prev_exit_to_depwait"] = r["depwait_med"] - prev_exit
        prev_exit = r["exit_max"]
        # slowest CTA: its last tile's accumulator-ready, partial-stored, ticket, reduced, epilogue-done
        slow = v[np.argmax(v[:, 4])]
        r["slowest"] = [round((int(slow[c]) - t0) / 1e3, 2) if slow[c] > 0 else None for c in (3, 8, 9, 10, 11, 4)]
        r["slowest_last_arriver"] = int(slow[12])
        rows.append({k: (round(v, 2) if isinstance(v, float) else v) for k, v in r.items()})
    span = rows[-1]["exit_max"] - rows[0]["start_min"]
    print(json.dumps({"op": "step-trace", "pdl": not a.no_pdl, "gemm_span_us": round(span, 1),
                      "first_layer": rows[:5], "layer_16": rows[80:85], "head": rows[-1]}))
    ctx.close()


if __name__ == "__main__":
    main()
