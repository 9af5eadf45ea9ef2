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

from .dllm import dllm_op_attention, dllm_op_gemm, dllm_op_gemm_timed, lib


def main(argv=None):
    ap = argparse.ArgumentParser()
    ap.add_argument("op", choices=("gemm", "attention", "gemm-sweep"))
    ap.add_argument("--M", type=int, default=24576)
    ap.add_argument("--N", type=int, default=32)
    ap.add_argument("--K", type=int, default=4096)
    ap.add_argument("--B", type=int, default=16)
    ap.add_argument("--T", type=int, default=64)
    ap.add_argument("--H", type=int, default=32)
    ap.add_argument("--P", type=int, default=4096)
    ap.add_argument("--reps", type=int, default=3)
    a = ap.parse_args(argv)
    lib()
    dev = torch.device("cuda:0")
    g = torch.Generator(device=dev)
    g.manual_seed(0)
    if a.op == "gemm-sweep":
        # kernel time vs weight rows: separates the fixed cost of a launch from the streaming rate
        rows = []
        for K in (4096, 12288):
            for M in (512, 1024, 2048, 4096, 8192, 12288, 24576, 49152, 126464):
                if M * K > 126464 * 4096:
                    continue
                W = (torch.randn(M, K, device=dev, generator=g) * 0.02).to(torch.bfloat16)
                X = torch.randn(a.N, K, device=dev, generator=g).to(torch.bfloat16)
                ms, _ = dllm_op_gemm_timed(W, X, M, a.N, K, a.reps)
                rows.append({"M": M, "N": a.N, "K": K, "us": ms * 1e3, "GBps": M * K * 2 / (ms * 1e-3) / 1e9})
                del W, X
        print(json.dumps({"op": "gemm-sweep", "rows": rows}))
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


if __name__ == "__main__":
    main()
