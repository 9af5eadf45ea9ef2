#!/usr/bin/env python
"""Benchmark of the block-wise diffusion-LLM denoising step on GB300.

Workload (default): one LLaDA-8B-shaped denoising step, bf16, batch 1: a
512-token uniform-random prompt prefilled into the prefix KV cache, then a
32-token window (the current block) with 24 positions masked; each step is
the whole hot path (embedding, 32 layers of RMSNorm / QKV+RoPE / attention /
O-proj / SwiGLU MLP, LM head with confidence and argmax, commit).  Weights are
random N(0, 0.02) drawn on the device; the data are synthetic.

Prints one JSON line.  `--impl reference` times the CPU oracle (the plain
fp32 C implementation) on this host's cores instead, on bounded samples of
the same step.
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import dllm_inputs as I  # noqa: E402

METRIC = "denoise steps/s & gen tokens/s at LLaDA-8B shape; % HBM / bf16 tensor roofline"
UNIT = "denoise steps/s"
SHAPE = dict(n_layers=32, d_model=4096, n_heads=32, head_dim=128, ffn=12288, vocab=126464, mask_id=126463,
             rope_base=500000.0)
WORKLOAD = dict(workload="llada8b_step_b1_p512_t32", model="LLaDA-8B-shaped (32L, d4096, 32x128, ffn12288, "
                "V126464), random N(0,0.02) bf16", batch=1, prompt=512, window=32, masked=24,
                commits_per_step=1, l2="inputs larger than L2 (15 GB of weights streamed per step)",
                seeds={"weights": I.SEED_WEIGHTS, "prompt": I.SEED_PROMPT})
LP, T, MASKED = 512, 32, 24


def _peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            p = json.load(f)
        return float(p["hbm_gbs"]), float(p["bf16_tflops"]), "measured"
    except Exception:
        return 6800.0, 1900.0, "fallback"


def _algorithmic_bytes(N):
    """Bytes each kind of launch must move at minimum (weights once, activations once)."""
    d, qd, F, V = 4096, 4096, 12288, 126464
    return {
        "qkv": 3 * qd * d * 2 + N * d * 2 + 3 * N * qd * 2,
        "oproj": d * qd * 2 + N * qd * 2 + 2 * N * d * 4,
        "gateup": 2 * F * d * 2 + N * d * 2 + N * F * 2,
        "down": d * F * 2 + N * F * 2 + 2 * N * d * 4,
        "head": V * d * 2 + N * d * 2 + (V // 128) * N * 12,
    }


def _attn_bytes(P, T_):
    return 2 * (P + T_) * 4096 * 2  # K and V rows of one layer (prefix + window), read once


class ClockSampler:
    """nvidia-smi clocks and throttle reasons sampled every 200 ms."""

    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.hw_slowdown,"
              "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
              "clocks_event_reasons.sw_power_cap")

    def __init__(self, uuid):
        self.uuid = uuid
        self.proc = None

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", self.uuid, f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "200"], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except Exception:
            self.proc = None

    def stop(self):
        if not self.proc:
            return None
        time.sleep(0.25)
        self.proc.terminate()
        try:
            out, _ = self.proc.communicate(timeout=5)
        except Exception:
            self.proc.kill()
            out, _ = self.proc.communicate()
        names = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap")
        sm, mx, reasons = [], [], set()
        for line in out.strip().splitlines():
            f = [x.strip() for x in line.split(",")]
            if len(f) < 7:
                continue
            try:
                sm.append(float(f[0]))
                mx.append(float(f[1]))
            except ValueError:
                continue
            for n, v in zip(names, f[3:7]):
                if v.lower().startswith("active"):
                    reasons.add(n)
        if not sm:
            return None
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx), "reasons": sorted(reasons),
                "samples": len(sm)}


def _dist_setup(args):
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    pg = None
    if world > 1:
        import torch.distributed as dist
        backend = "nccl" if args.impl == "ours" else "gloo"
        dist.init_process_group(backend)
        pg = dist
    return world, rank, local, pg


def _max_over_ranks(value, pg, device=None):
    if pg is None:
        return value
    import torch
    t = torch.tensor([value], dtype=torch.float64, device=device)
    pg.all_reduce(t, op=pg.ReduceOp.MAX)
    return float(t.item())


def _barrier(pg, device=None):
    if pg is None:
        return
    if device is not None:
        pg.barrier(device_ids=[device.index])
    else:
        pg.barrier()


# ---------------------------------------------------------------------------------------- oracle leg
class OracleSample:
    """A bounded sample of one step on the CPU oracle: `layers` transformer
    layers of the 32-token window over a 512-token prefix, and the LM head over
    1/`head_div` of the vocabulary rows, both scaled to the full step."""

    def __init__(self, layers, head_div):
        import numpy as np
        import oracle as O

        O.build()
        self.O = O
        self.layers, self.head_div = layers, head_div
        self.lmodel = O.Model(O.OracleConfig(**dict(SHAPE, n_layers=layers)), gen_layers=layers, gen_head=False)
        hv = SHAPE["vocab"] // head_div
        self.hmodel = O.Model(O.OracleConfig(**dict(SHAPE, n_layers=1, vocab=hv, mask_id=hv - 1)), gen_layers=0,
                              gen_head=True)
        rng = np.random.default_rng(I.SEED_KV)
        self.pk = rng.standard_normal((layers, LP, 4096), dtype=np.float32)
        self.pv = rng.standard_normal((layers, LP, 4096), dtype=np.float32)
        self.tok = I.uniform_prompt(T, SHAPE["vocab"], SHAPE["mask_id"], seed=7)
        self.htok = self.tok % (hv - 1)
        self.pos = np.arange(LP, LP + T, dtype=np.int32)
        self.desc = (f"{layers} of 32 layers (32-token window over a 512-token prefix) scaled x{32 / layers:g}, "
                     f"plus the LM head over 1/{head_div} of the vocabulary scaled x{head_div}")

    def seconds_per_step(self):
        O = self.O
        t0 = time.perf_counter()
        O.forward(self.lmodel, self.tok, self.pos, prefix_k=self.pk, prefix_v=self.pv, logits=False,
                  n_layers_run=self.layers)
        t1 = time.perf_counter()
        O.forward(self.hmodel, self.htok, self.pos, logits=True, n_layers_run=0)
        t2 = time.perf_counter()
        return (t1 - t0) * 32.0 / self.layers + (t2 - t1) * self.head_div, t2 - t0


def run_reference(args):
    world, rank, local, pg = _dist_setup(args)
    if rank != 0:
        return 0
    cores = os.cpu_count()
    sample = OracleSample(1, 32)
    for _ in range(min(args.warmup, 1)):
        sample.seconds_per_step()
    est, cpu = 0.0, 0.0
    for _ in range(args.steps):
        e, c = sample.seconds_per_step()
        est += e
        cpu += c
    value = args.steps / est
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": 1, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": 1000.0 * est / args.steps, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f32", "data": "synthetic", "config": WORKLOAD,
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": cores, "kind": "oracle",
                         "sample": "each step: " + sample.desc + f" ({cpu / args.steps:.2f} s of CPU time)"},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)
    return 0


# ---------------------------------------------------------------------------------------- GPU leg
def run_ours(args):
    import numpy as np
    import torch

    world, rank, local, pg = _dist_setup(args)
    torch.cuda.set_device(local)
    device = torch.device("cuda", local)
    from paper_2606_13740_gb300 import COMMITTED, MASKED, Config, Context, Sched

    cfg = Config(max_batch=1, max_ctx=LP + T, max_window=LP, **SHAPE)
    ctx = Context(cfg)
    if args.no_pdl or args.full_smem:
        ctx.dllm_set_debug((4 if args.no_pdl else 0) | (8 if args.full_smem else 0))
    stream = ctx.stream  # the context's own stream: events and kernels share it
    sched = Sched(steps_per_block=MASKED)
    prompt = I.uniform_prompt(LP, cfg.vocab, cfg.mask_id, seed=I.SEED_PROMPT + rank)
    ctx.dllm_prefill(sched, prompt, T)
    ctx.dllm_begin_block()
    tok, st, _ = ctx.dllm_get_state()
    win = np.arange(LP, LP + T)
    tok[0, win] = I.uniform_prompt(T, cfg.vocab, cfg.mask_id, seed=7)
    st[0, win] = COMMITTED
    m = win[I.masked_positions(T, MASKED)]
    tok[0, m], st[0, m] = cfg.mask_id, MASKED
    ctx.dllm_set_state(tok, st)  # every step starts from this window (rewound per block)

    state = {"in_block": 0, "rewinds": 0}

    def step():
        if state["in_block"] == MASKED:
            ctx.dllm_rewind_block()
            state["in_block"] = 0
            state["rewinds"] += 1
        ctx.dllm_denoise_step(want_out=False)
        state["in_block"] += 1

    for _ in range(max(args.warmup, 3)):
        step()
    torch.cuda.synchronize()
    launches = ctx.dllm_launches_per_step()

    sampler = ClockSampler(str(torch.cuda.get_device_properties(device).uuid))
    if not sampler.uuid.startswith("GPU-"):
        sampler.uuid = "GPU-" + sampler.uuid
    _barrier(pg, device)
    torch.cuda.synchronize()
    sampler.start()
    time.sleep(0.3)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    state["rewinds"] = 0
    e0.record(stream)
    for _ in range(args.steps):
        step()
    e1.record(stream)
    torch.cuda.synchronize()
    clocks = sampler.stop()
    _barrier(pg, device)
    ms = e0.elapsed_time(e1)
    rewinds = state["rewinds"]
    ms_max = _max_over_ranks(ms, pg, device)
    ms_per_step = ms_max / args.steps
    value = world * args.steps / (ms_max / 1000.0)

    # per-kernel durations over the same steps, with events captured into the step graph
    ctx.dllm_set_profile(1)
    nprof = min(args.steps, 48)
    for _ in range(nprof):
        step()
    prof, psteps = ctx.dllm_get_profile()
    ctx.dllm_set_profile(0)

    # end to end through the public API with host buffers (pinned), copies inside the timed region
    tok_h = torch.from_numpy(tok.copy()).pin_memory().numpy()
    st_h = torch.from_numpy(st.copy()).pin_memory().numpy()
    ne2e = max(10, min(args.steps, 100))
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    for _ in range(ne2e):
        ctx.dllm_set_state(tok_h, st_h)
        ctx.dllm_denoise_step(want_out=True)
        out_tok, out_st, out_kv = ctx.dllm_get_state()
    e2e_s = time.perf_counter() - t0
    e2e_s = _max_over_ranks(e2e_s, pg, device)
    n_pos = LP + T
    h2d = n_pos * 5
    d2h = n_pos * 5 + 4 + 8 * 4

    hbm, bf16, peak_src = _peaks()
    algo = _algorithmic_bytes(T)
    # dominant kernel: the chained projections of a layer (output, gate/up, down, then the next
    # layer's QKV; the last layer's chain ends with the LM head instead)
    layer = prof["layer"]
    n_chain = max(1, psteps * layer["launches_per_step"])
    chain_ms = layer["ms_total"] / n_chain
    per_layer = algo["oproj"] + algo["gateup"] + algo["down"]
    chain_bytes = (31 * (per_layer + algo["qkv"]) + per_layer + algo["head"]) / 32  # average launch
    achieved = chain_bytes / (chain_ms * 1e-3) / 1e9
    step_bytes = 32 * (algo["qkv"] + algo["oproj"] + algo["gateup"] + algo["down"] + _attn_bytes(LP, T)) + algo["head"]
    step_ach = step_bytes / (ms_per_step * 1e-3) / 1e9
    gemm_ms = (prof["qkv"]["ms_total"] + layer["ms_total"]) / max(1, psteps)
    gemm_bytes = 32 * (algo["qkv"] + algo["oproj"] + algo["gateup"] + algo["down"]) + algo["head"]
    traffic = None
    try:  # DRAM bytes of one layer-chain launch from an ncu capture of this exact source
        with open(os.path.join(ROOT, "profiles", "chain_layer_traffic.json")) as f:
            tr = json.load(f)
        if tr.get("source_hash") == _kernel_hash():
            traffic = tr["dram_bytes_per_launch"]
    except Exception:
        pass
    line = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
        "warmup": max(args.warmup, 3), "ms_per_step": ms_per_step, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "bf16", "data": "synthetic", "config": WORKLOAD,
        "parallelism": "replicas" if world > 1 else "single-gpu",
        "gen_tokens_per_s": value * WORKLOAD["commits_per_step"],
        "roofline": {"kernel": "k_chain (one layer: output, gate/up, down and next-QKV projections, "
                               "436 MB of weights per launch)", "bound": "hbm",
                     "achieved": achieved, "peak": hbm, "unit": "GB/s", "frac": achieved / hbm,
                     "traffic": traffic, "peak_source": peak_src,
                     "algorithmic_bytes_per_launch": chain_bytes, "avg_launch_ms": chain_ms},
        "step_roofline": {"bound": "hbm", "algorithmic_bytes_per_step": step_bytes, "achieved": step_ach,
                          "peak": hbm, "unit": "GB/s", "frac": step_ach / hbm,
                          "gemm_achieved": gemm_bytes / (gemm_ms * 1e-3) / 1e9},
        "kernel_ms_per_step": {k: v["ms_total"] / max(1, psteps) for k, v in prof.items()},
        "e2e": {"value": world * ne2e / e2e_s, "unit": UNIT, "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h},
        "gpu_launches": launches * args.steps + rewinds,
        "clocks": clocks,
    }
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        try:
            # the sample repeated until it has taken at least 10 s (at most 16 times), after one
            # untimed pass; the step estimate is the mean over the repetitions
            sample = OracleSample(4, 8)
            sample.seconds_per_step()
            per_sum, cpu, reps = 0.0, 0.0, 0
            while cpu < 10.0 and reps < 16:
                p, c = sample.seconds_per_step()
                per_sum += p
                cpu += c
                reps += 1
            per = per_sum / reps
            line["cpu_baseline"] = {"value": 1.0 / per, "unit": UNIT, "cores": os.cpu_count(), "kind": "oracle",
                                    "sample": sample.desc + f", repeated {reps} times ({cpu:.1f} s of CPU time)"}
        except Exception as exc:  # reported, not fatal
            line["cpu_baseline"] = {"value": None, "unit": UNIT, "cores": os.cpu_count(), "kind": "oracle",
                                    "sample": f"failed: {exc}"}
    ctx.close()
    if rank == 0:
        print(json.dumps(line), flush=True)
    if pg is not None:
        pg.destroy_process_group()
    return 0


def _kernel_hash():
    import hashlib
    h = hashlib.sha256()
    csrc = os.path.join(ROOT, "paper_2606_13740_gb300", "csrc")
    for name in sorted(os.listdir(csrc)):
        if name.startswith("gemm") or name.endswith(".cuh") or name == "internal.h":
            with open(os.path.join(csrc, name), "rb") as f:
                h.update(f.read())
    return h.hexdigest()[:16]


def main(argv=None):
    ap = argparse.ArgumentParser(description=__doc__.splitlines()[0])
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=300)
    ap.add_argument("--warmup", type=int, default=10)
    ap.add_argument("--impl", choices=("ours", "reference"), default="ours")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-pdl", action="store_true", help="launch kernels without programmatic dependent launch")
    ap.add_argument("--full-smem", action="store_true", help="one 227 KB projection CTA per SM (no co-residency)")
    args = ap.parse_args(argv)
    if args.impl == "reference":
        return run_reference(args)
    return run_ours(args)


if __name__ == "__main__":
    sys.exit(main())
