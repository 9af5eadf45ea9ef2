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
    ap.add_argument("op", choices=("gemm", "attention", "gemm-sweep", "gemm-trace", "step-trace", "step-small"))
    ap.add_argument("--M", type=int, default=24576)
    ap.add_argument("--N", type=int, default=32)
    ap.add_argument("--K", type=int, default=4096)
    ap.add_argument("--B", type=int, default=16)
    ap.add_argument("--T", type=int, default=64)
    ap.add_argument("--H", type=int, default=32)
    ap.add_argument("--P", type=int, default=4096)
    ap.add_argument("--reps", type=int, default=3)
    ap.add_argument("--dump", default="", help="gemm-trace: write every CTA's timeline to this JSON file")
    ap.add_argument("--no-pdl", action="store_true")
    ap.add_argument("--debug", type=int, default=0, help="step-trace: extra dllm_set_debug flags")
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
    cfg = Config(max_batch=1, max_ctx=544, max_window=512, **shape)
    ctx = Context(cfg)
    flags = 16 | (4 if a.no_pdl else 0) | a.debug
    ctx.dllm_set_debug(flags)
    rng = np.random.default_rng(1)
    prompt = rng.integers(0, cfg.vocab - 1, 512).astype(np.int32)
    ctx.dllm_prefill(Sched(steps_per_block=24), prompt, 32)
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
