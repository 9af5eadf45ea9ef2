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

from .dllm import dllm_op_attention, dllm_op_gemm, lib


def main(argv=None):
    ap = argparse.ArgumentParser()
    ap.add_argument("op", choices=("gemm", "attention", "step-small", "step-small-b16"))
    ap.add_argument("--M", type=int, default=24576)
    ap.add_argument("--N", type=int, default=32)
    ap.add_argument("--K", type=int, default=4096)
    ap.add_argument("--B", type=int, default=16)
    ap.add_argument("--T", type=int, default=64, help="attention: window tokens")
    ap.add_argument("--H", type=int, default=32)
    ap.add_argument("--P", type=int, default=4096)
    ap.add_argument("--reps", type=int, default=3)
    ap.add_argument("--weight-bits", type=int, default=16, help="step-small: 16 (bf16) or 4 (4-bit block format)")
    a = ap.parse_args(argv)
    lib()
    if a.op == "step-small":
        step_small(a)
        return
    if a.op == "step-small-b16":
        step_small_b16(a)
        return
    dev = torch.device("cuda:0")
    g = torch.Generator(device=dev)
    g.manual_seed(0)
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
    the small case for ncu captures of the step's kernels (--weight-bits 4: the projections in
    the 4-bit block format)."""
    import numpy as np

    from .dllm import Config, Context, Sched

    shape = dict(n_layers=2, d_model=4096, n_heads=32, head_dim=128, ffn=12288, vocab=126464, mask_id=126463,
                 rope_base=500000.0)
    ctx = Context(Config(max_batch=1, max_ctx=544, max_window=512, weight_bits=a.weight_bits, **shape))
    rng = np.random.default_rng(1)
    ctx.dllm_prefill(Sched(steps_per_block=24), rng.integers(0, 126463, 512).astype(np.int32), 32)
    ctx.dllm_begin_block()
    for _ in range(a.reps):
        ctx.dllm_denoise_step(want_out=False)
    ctx.dllm_sync()
    ctx.close()
    print(json.dumps({"op": "step-small", "steps": a.reps}))



def step_small_b16(a):
    """A few batch-16 denoising steps of a 2-layer model at the LLaDA-8B width: synthetic prefix
    K/V of 4096 positions per sequence, a 64-token window with 32 masked (about 6 GB on the
    device): the small case for ncu captures of the batch-16 step's kernels."""
    import numpy as np

    import dllm_inputs as I

    from .dllm import COMMITTED, MASKED, Config, Context, Sched

    shape = dict(n_layers=2, d_model=4096, n_heads=32, head_dim=128, ffn=12288, vocab=126464, mask_id=126463,
                 rope_base=500000.0)
    B, P, T = 16, 4096, 64
    ctx = Context(Config(max_batch=B, max_ctx=P + T, max_window=T, **shape))
    sched = Sched(steps_per_block=32, spec_trigger=32, spec_blocks=1)
    ctx.dllm_set_prefix_kv_random(sched, B, P, T, I.SEED_KV)
    ctx.dllm_begin_block()
    tok, st, _ = ctx.dllm_get_state()
    win = np.arange(P, P + T)
    tok[:, win] = I.zipf_ids((B, T), shape["vocab"], shape["mask_id"])
    st[:, win] = COMMITTED
    for b in range(B):
        m = win[I.masked_positions(T, 32, seed=I.SEED_PROMPT + 100 + b)]
        tok[b, m], st[b, m] = shape["mask_id"], MASKED
    ctx.dllm_set_state(tok, st)
    for _ in range(a.reps):
        ctx.dllm_rewind_block()
        ctx.dllm_denoise_step(want_out=False)
    ctx.dllm_sync()
    ctx.close()
    print(json.dumps({"op": "step-small-b16", "steps": a.reps}))


if __name__ == "__main__":
    main()
