#!/usr/bin/env python
"""Benchmark of the block-wise diffusion-LLM denoising path on GB300.

Workload (default, `llada8b_step_b1_p512_t32`): one LLaDA-8B-shaped denoising
step, bf16, batch 1: a 512-token uniform-random prompt prefilled into the
prefix KV cache, then a 32-token window (the current block) with 24 positions
masked; each step is the whole hot path (embedding, 32 layers of RMSNorm /
QKV+RoPE / attention / O-proj / SwiGLU MLP, LM head with confidence and argmax,
commit).  Weights are random N(0, 0.02) drawn on the device; the data are
synthetic.

Other workloads (`--workload`, one JSON line each, same schema):
  llada8b_step_b1_p512_t32_q4      the default step with the projections and the LM head in
                                   the 4-bit block format of the paper's Q4_0 weights
  llada8b_step_b16_p4096_t64       batched serving step: 16 sequences, synthetic
                                   4096-position prefix KV each, 64-token window
                                   (current block + one speculative block), 32
                                   masked, Zipf(1.1) ids
  llada8b_gen_p256_g128            whole generation: 256-token prompt, 4 blocks of
                                   32, 32 steps per block, one commit per step
  llada8b_gen_spec_rev_p1024_g256  whole generation with multi-block speculation
                                   (window 96 once <= 8 masked) and revision
                                   (re-mask below 0.5)
  llada8b_gen_*                    the same generation with the paper's other
                                   decoding options (threshold commit, sparse cache
                                   refresh, continuous sliding, adaptive lookahead)
  llada8b_window_sweep_b1_p512     step time against the window length
  all                              every workload above, one line each

Prints one JSON line per workload.  `--impl reference` times the CPU oracle
(the plain fp32 C implementation) on this host's cores instead, on bounded
samples of the same step.
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
GEN_UNIT = "generated tokens/s"
SHAPE = dict(n_layers=32, d_model=4096, n_heads=32, head_dim=128, ffn=12288, vocab=126464, mask_id=126463,
             rope_base=500000.0)
MODEL = ("LLaDA-8B-shaped (32L, d4096, 32x128, ffn12288, V126464), random N(0,0.02) bf16")
SEEDS = {"weights": I.SEED_WEIGHTS, "prompt": I.SEED_PROMPT}
WORKLOAD = dict(workload="llada8b_step_b1_p512_t32", model=MODEL, batch=1, prompt=512, window=32, masked=24,
                commits_per_step=1, l2="inputs larger than L2 (15 GB of weights streamed per step)", seeds=SEEDS)
LP, T, MASKED = 512, 32, 24

# whole-generation workloads: (prompt, generated tokens, schedule keywords, what it exercises)
GENERATIONS = {
    "llada8b_gen_p256_g128": (256, 128, dict(steps_per_block=32),
                              "4 blocks of 32, 32 steps per block, one commit per step (Sec. 2.1)"),
    "llada8b_gen_spec_rev_p1024_g256": (
        1024, 256, dict(steps_per_block=32, spec_trigger=8, spec_blocks=2, theta_remask=0.5, remask_max=1),
        "8 blocks; window 96 (2 speculative blocks) once <= 8 positions are masked (Sec. 3.2); committed "
        "tokens re-masked below confidence 0.5, at most 1 per step (Sec. 3.3)"),
    "llada8b_gen_threshold_p256_g128": (
        256, 128, dict(steps_per_block=32, commit_mode=1, theta_visible=0.7, theta_stable=0.9),
        "staged token stabilization's threshold commit, 0.7 visible / 0.9 stable (Sec. 3.3); random weights "
        "stay below 0.7, so every step takes the single-position fallback"),
    "llada8b_gen_scr32_p256_g128": (256, 128, dict(steps_per_block=32, scr_rows=32),
                                    "sparse cache refresh of 32 visible prefix positions per step (Sec. 3.3)"),
    "llada8b_gen_slide_p256_g128": (256, 128, dict(steps_per_block=32, slide=1),
                                    "continuous sliding of the window along the commit frontier (Sec. 3.2)"),
    "llada8b_gen_slide_lookahead_p1024_g256": (
        1024, 256, dict(steps_per_block=32, slide=1, spec_trigger=8, spec_blocks=2, theta_remask=0.5,
                        remask_max=1),
        "continuous sliding with two lookahead blocks and revision (Sec. 3.2, 3.3)"),
    "llada8b_gen_adaptive_p1024_g256": (
        1024, 256, dict(steps_per_block=32, spec_trigger=8, spec_blocks=2, theta_remask=0.5, remask_max=1,
                        spec_allowance=0.2),
        "adaptive lookahead from the window sweep's step latencies, allowance 0.2 (Sec. 3.2)"),
}
STEP_B16 = "llada8b_step_b16_p4096_t64"
STEP_Q4 = "llada8b_step_b1_p512_t32_q4"
SWEEP = "llada8b_window_sweep_b1_p512"
ALL = [WORKLOAD["workload"], STEP_Q4, STEP_B16, SWEEP, *GENERATIONS]


def _peaks():
    """(HBM GB/s, bf16 TFLOP/s burst, sustained, source)."""
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            p = json.load(f)
        return (float(p["hbm_gbs"]), float(p["bf16_tflops"]),
                float(p.get("bf16_tflops_sustained", p["bf16_tflops"])), "measured")
    except Exception:
        return 6800.0, 1900.0, 1700.0, "fallback"


def _algorithmic_bytes(N, wb=2.0):
    """Bytes each kind of launch must move at minimum (weights once at wb bytes per weight,
    activations once)."""
    d, qd, F, V = 4096, 4096, 12288, 126464
    return {
        "qkv": 3 * qd * d * wb + N * d * 2 + 3 * N * qd * 2,
        "oproj": d * qd * wb + N * qd * 2 + 2 * N * d * 4,
        "gateup": 2 * F * d * wb + N * d * 2 + N * F * 2,
        "down": d * F * wb + N * F * 2 + 2 * N * d * 4,
        "head": V * d * wb + N * d * 2 + (V // 128) * N * 12,
    }


Q4_BYTES = 0.5 + 2.0 / 32  # 4-bit code plus a bf16 scale per block of 32: 4.5 bits per weight


def _attn_bytes(P, T_):
    return 2 * (P + T_) * 4096 * 2  # K and V rows of one layer (prefix + window), read once


def _step_bytes(P, T_, wb=2.0):
    a = _algorithmic_bytes(T_, wb)
    return 32 * (a["qkv"] + a["oproj"] + a["gateup"] + a["down"] + _attn_bytes(P, T_)) + a["head"]


def _layer_flops(N):
    d, F = 4096, 12288
    return 2 * N * (4 * d * d + 3 * d * F)


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
    """A bounded sample of one step on the CPU oracle: `layers` transformer layers of one
    sequence's T-token window over a P-token prefix (synthetic prefix K/V), and the LM head over
    1/`head_div` of the vocabulary rows for `head_rows` of the window's rows, all scaled to the
    full step (32 layers, `batch` sequences, every row of the head)."""

    def __init__(self, layers, head_div, P=LP, T_=T, batch=1, head_rows=None, weight_bits=16):
        import numpy as np
        import oracle as O

        O.build()
        self.O = O
        self.layers, self.head_div, self.batch = layers, head_div, batch
        self.head_rows = T_ if head_rows is None else head_rows
        self.lmodel = O.Model(O.OracleConfig(**dict(SHAPE, n_layers=layers, weight_bits=weight_bits)),
                              gen_layers=layers, gen_head=False)
        hv = SHAPE["vocab"] // head_div
        self.hmodel = O.Model(O.OracleConfig(**dict(SHAPE, n_layers=1, vocab=hv, mask_id=hv - 1,
                                                    weight_bits=weight_bits)), gen_layers=0, gen_head=True)
        rng = np.random.default_rng(I.SEED_KV)
        self.pk = rng.standard_normal((layers, P, 4096), dtype=np.float32)
        self.pv = rng.standard_normal((layers, P, 4096), dtype=np.float32)
        self.tok = I.uniform_prompt(T_, SHAPE["vocab"], SHAPE["mask_id"], seed=7)
        self.htok = self.tok[:self.head_rows] % (hv - 1)
        self.pos = np.arange(P, P + T_, dtype=np.int32)
        self.scale_head = head_div * batch * T_ / self.head_rows
        self.desc = (f"{layers} of 32 layers ({T_}-token window over a {P}-token prefix) scaled "
                     f"x{32 * batch / layers:g}, plus the LM head over 1/{head_div} of the vocabulary for "
                     f"{self.head_rows} rows scaled x{self.scale_head:g}; extrapolated to the full step")

    def seconds_per_step(self):
        O = self.O
        t0 = time.perf_counter()
        O.forward(self.lmodel, self.tok, self.pos, prefix_k=self.pk, prefix_v=self.pv, logits=False,
                  n_layers_run=self.layers)
        t1 = time.perf_counter()
        O.forward(self.hmodel, self.htok, self.pos[:self.head_rows], logits=True, n_layers_run=0)
        t2 = time.perf_counter()
        return (t1 - t0) * 32.0 * self.batch / self.layers + (t2 - t1) * self.scale_head, t2 - t0


def _cpu_baseline(sample, unit, to_value, min_cpu_s=10.0):
    """The sample repeated until it has taken min_cpu_s (at most 16 times), after one untimed pass;
    to_value maps the mean estimated seconds per step to the line's unit."""
    try:
        sample.seconds_per_step()
        per_sum, cpu, reps = 0.0, 0.0, 0
        while cpu < min_cpu_s and reps < 16:
            p, c = sample.seconds_per_step()
            per_sum += p
            cpu += c
            reps += 1
        per = per_sum / reps
        return {"value": to_value(per), "unit": unit, "cores": os.cpu_count(), "kind": "oracle",
                "extrapolated": True, "seconds_per_step_estimate": per,
                "sample": sample.desc + f", repeated {reps} times ({cpu:.1f} s of CPU time)"}
    except Exception as exc:  # reported, not fatal
        return {"value": None, "unit": unit, "cores": os.cpu_count(), "kind": "oracle", "sample": f"failed: {exc}"}


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
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": cores, "kind": "oracle", "extrapolated": True,
                         "sample": "each step: " + sample.desc + f" ({cpu / args.steps:.2f} s of CPU time); "
                                   "ms_per_step is the extrapolated full step, not the sample's own time"},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)
    return 0


# ---------------------------------------------------------------------------------------- GPU leg
class Timed:
    """Clock sampling, barrier and CUDA events around a timed region on one stream."""

    def __init__(self, torch, device, stream, pg):
        self.torch, self.device, self.stream, self.pg = torch, device, stream, pg
        uuid = str(torch.cuda.get_device_properties(device).uuid)
        self.sampler = ClockSampler(uuid if uuid.startswith("GPU-") else "GPU-" + uuid)

    def __enter__(self):
        torch = self.torch
        _barrier(self.pg, self.device)
        torch.cuda.synchronize()
        self.sampler.start()
        time.sleep(0.3)
        self.e0, self.e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        self.t0 = time.perf_counter()
        self.e0.record(self.stream)
        return self

    def __exit__(self, *exc):
        self.e1.record(self.stream)
        self.torch.cuda.synchronize()
        self.wall = time.perf_counter() - self.t0
        self.clocks = self.sampler.stop()
        _barrier(self.pg, self.device)
        self.ms = _max_over_ranks(self.e0.elapsed_time(self.e1), self.pg, self.device)
        return False


def _chain_roofline(prof, psteps, per_launch_units, unit, peak, peak_source, bound, kernel):
    """Dominant kernel: the layer chains (output, gate/up, down, next QKV or the head), the average
    launch's algorithmic work over its average duration from events in the step graph."""
    layer = prof["layer"]
    n_chain = max(1, psteps * layer["launches_per_step"])
    chain_ms = layer["ms_total"] / n_chain
    achieved = per_launch_units / (chain_ms * 1e-3) / (1e9 if unit == "GB/s" else 1e12)
    return {"kernel": kernel, "bound": bound, "achieved": achieved, "peak": peak, "unit": unit,
            "frac": achieved / peak, "traffic": None, "peak_source": peak_source,
            ("algorithmic_bytes_per_launch" if unit == "GB/s" else "algorithmic_flops_per_launch"): per_launch_units,
            "avg_launch_ms": chain_ms}


def run_step_b1(args, env, q4=False):
    import numpy as np
    torch, device, world, rank, pg = env["torch"], env["device"], env["world"], env["rank"], env["pg"]
    from paper_2606_13740_gb300 import COMMITTED, MASKED, Config, Context, Sched

    cfg = Config(max_batch=1, max_ctx=LP + T, max_window=LP, weight_bits=4 if q4 else 16, **SHAPE)
    wb = Q4_BYTES if q4 else 2.0
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
    state["rewinds"] = 0
    with Timed(torch, device, stream, pg) as tm:
        for _ in range(args.steps):
            step()
    rewinds = state["rewinds"]
    ms_per_step = tm.ms / args.steps
    value = world * args.steps / (tm.ms / 1000.0)

    # per-kernel durations over the same steps, with events captured into the step graph
    ctx.dllm_set_profile(1)
    for _ in range(min(args.steps, 48)):
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
        ctx.dllm_get_state()
    e2e_s = _max_over_ranks(time.perf_counter() - t0, pg, device)
    n_pos = LP + T

    hbm, bf16, bf16_sus, peak_src = env["peaks"]
    algo = _algorithmic_bytes(T, wb)
    per_layer = algo["oproj"] + algo["gateup"] + algo["down"]
    chain_bytes = (31 * (per_layer + algo["qkv"]) + per_layer + algo["head"]) / 32  # average launch
    roof = _chain_roofline(prof, psteps, chain_bytes, "GB/s", hbm, peak_src, "hbm",
                           "k_chain (one layer: output, gate/up, down and next-QKV projections, "
                           + ("123 MB of 4-bit weights per launch, expanded to bf16 in shared memory)"
                              if q4 else "436 MB of weights per launch)"))
    if not q4:
        try:  # DRAM bytes of one layer-chain launch from an ncu capture of this exact source
            with open(os.path.join(ROOT, "profiles", "chain_layer_traffic.json")) as f:
                tr = json.load(f)
            if tr.get("source_hash") == _kernel_hash():
                roof["traffic"] = tr["dram_bytes_per_launch"]
        except Exception:
            pass
    step_bytes = _step_bytes(LP, T, wb)
    step_ach = step_bytes / (ms_per_step * 1e-3) / 1e9
    gemm_ms = (prof["qkv"]["ms_total"] + prof["layer"]["ms_total"]) / max(1, psteps)
    gemm_bytes = 32 * (algo["qkv"] + algo["oproj"] + algo["gateup"] + algo["down"]) + algo["head"]
    line = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
        "warmup": max(args.warmup, 3), "ms_per_step": ms_per_step, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": dict(WORKLOAD, workload=STEP_Q4, weights="4-bit block format (Q4_0-style: 32 weights per "
                       "bf16 scale, codes 0..15 for d*(q-8)), 4.5 bits per weight; bf16 arithmetic") if q4 else WORKLOAD,
        "parallelism": "replicas" if world > 1 else "single-gpu",
        "gen_tokens_per_s": value * WORKLOAD["commits_per_step"],
        "roofline": roof,
        "step_roofline": {"bound": "hbm", "algorithmic_bytes_per_step": step_bytes, "achieved": step_ach,
                          "peak": hbm, "unit": "GB/s", "frac": step_ach / hbm,
                          "gemm_achieved": gemm_bytes / (gemm_ms * 1e-3) / 1e9},
        "kernel_ms_per_step": {k: v["ms_total"] / max(1, psteps) for k, v in prof.items()},
        "e2e": {"value": world * ne2e / e2e_s, "unit": UNIT, "h2d_bytes_per_step": n_pos * 5,
                "d2h_bytes_per_step": n_pos * 5 + 4 + 8 * 4},
        "gpu_launches": launches * args.steps + rewinds,
        "clocks": tm.clocks,
    }
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        line["cpu_baseline"] = _cpu_baseline(OracleSample(4, 8, weight_bits=4 if q4 else 16), UNIT,
                                             lambda s: 1.0 / s)
    ctx.close()
    return line


def run_step_b16(args, env):
    import numpy as np
    torch, device, world, rank, pg = env["torch"], env["device"], env["world"], env["rank"], env["pg"]
    from paper_2606_13740_gb300 import COMMITTED, MASKED, Config, Context, Sched

    B, P, Tw, M = 16, 4096, 64, 32
    cfg = Config(max_batch=B, max_ctx=P + Tw, max_window=Tw, **SHAPE)
    ctx = Context(cfg)
    sched = Sched(steps_per_block=32, spec_trigger=32, spec_blocks=1)
    ctx.dllm_set_prefix_kv_random(sched, B, P, Tw, I.SEED_KV + rank)
    ctx.dllm_begin_block()
    tok, st, _ = ctx.dllm_get_state()
    win = np.arange(P, P + Tw)
    tok[:, win] = I.zipf_ids((B, Tw), cfg.vocab, cfg.mask_id, seed=I.SEED_ZIPF + rank)
    st[:, win] = COMMITTED
    for b in range(B):
        m = win[I.masked_positions(Tw, M, seed=I.SEED_PROMPT + 100 + b)]
        tok[b, m], st[b, m] = cfg.mask_id, MASKED
    ctx.dllm_set_state(tok, st)

    def step():
        ctx.dllm_rewind_block()
        ctx.dllm_denoise_step(want_out=False)

    for _ in range(max(args.warmup, 3)):
        step()
    torch.cuda.synchronize()
    launches = ctx.dllm_launches_per_step()
    window = ctx.dllm_window()
    steps = max(3, min(args.steps, 40))
    with Timed(torch, device, ctx.stream, pg) as tm:
        for _ in range(steps):
            step()
    ms_per_step = tm.ms / steps
    value = world * steps / (tm.ms / 1000.0)
    ctx.dllm_set_profile(1)
    for _ in range(min(steps, 8)):
        step()
    prof, psteps = ctx.dllm_get_profile()
    ctx.dllm_set_profile(0)
    tok_h = torch.from_numpy(tok.copy()).pin_memory().numpy()
    st_h = torch.from_numpy(st.copy()).pin_memory().numpy()
    ne2e = max(5, min(steps, 20))
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    for _ in range(ne2e):
        ctx.dllm_set_state(tok_h, st_h)
        ctx.dllm_denoise_step(want_out=True)
        ctx.dllm_get_state()
    e2e_s = _max_over_ranks(time.perf_counter() - t0, pg, device)

    hbm, bf16, bf16_sus, peak_src = env["peaks"]
    N = B * Tw
    head_flops = 2 * N * cfg.vocab * cfg.d_model
    chain_flops = (31 * _layer_flops(N) + _layer_flops(N) + head_flops) / 32  # average layer-chain launch
    roof = _chain_roofline(prof, psteps, chain_flops, "TFLOP/s", bf16_sus, peak_src + " (sustained: the kernel "
                           "runs inside a 20 ms step)", "tensor",
                           "k_chain (one layer: output, gate/up, down and next-QKV projections over 1024 tokens)")
    attn_ms = prof["attn"]["ms_total"] / max(1, psteps * prof["attn"]["launches_per_step"])
    attn_bytes = B * _attn_bytes(P, Tw)
    attn_ach = attn_bytes / (attn_ms * 1e-3) / 1e9
    step_flops = 32 * _layer_flops(N) + head_flops + B * 32 * 4 * Tw * (P + Tw) * cfg.d_model
    step_bytes = 32 * (B * _attn_bytes(P, Tw)) + 14.995e9
    gemm_ms = 32 * roof["avg_launch_ms"] + prof["qkv"]["ms_total"] / max(1, psteps)
    line = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": steps,
        "warmup": max(args.warmup, 3), "ms_per_step": ms_per_step, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": dict(workload=STEP_B16, model=MODEL, batch=B, prefix=P, window=Tw, masked_per_sequence=M,
                       ids="Zipf(1.1)", prefix_kv="synthetic N(0,1) from the seeded generator (no prefill)",
                       l2="inputs larger than L2 (15 GB of weights and 34 GB of K/V per step)",
                       seeds=dict(SEEDS, kv=I.SEED_KV, zipf=I.SEED_ZIPF)),
        "sequence_steps_per_s": value * B,
        "window": window,
        "roofline": roof,
        "attn_roofline": {"kernel": "k_attn_tc (tcgen05 split-KV attention, 16 x 32 heads x 64 queries x "
                                    f"{P + Tw} keys)", "bound": "hbm", "achieved": attn_ach, "peak": hbm,
                          "unit": "GB/s", "frac": attn_ach / hbm, "algorithmic_bytes_per_launch": attn_bytes,
                          "avg_launch_ms": attn_ms, "peak_source": peak_src},
        "step_roofline": {"algorithmic_flops_per_step": step_flops, "algorithmic_bytes_per_step": step_bytes,
                          "roofline_ms": 1e3 * (32 * _layer_flops(N) + head_flops) / (bf16 * 1e12)
                          + 1e3 * 32 * B * _attn_bytes(P, Tw) / (hbm * 1e9),
                          "gemm_ms_per_step": gemm_ms, "achieved_tflops": step_flops / (ms_per_step * 1e-3) / 1e12},
        "kernel_ms_per_step": {k: v["ms_total"] / max(1, psteps) for k, v in prof.items()},
        "e2e": {"value": world * ne2e / e2e_s, "unit": UNIT, "h2d_bytes_per_step": B * (P + Tw) * 5,
                "d2h_bytes_per_step": B * (P + Tw) * 5 + 4 * B + 8 * 4},
        "gpu_launches": (launches + 1) * steps,
        "clocks": tm.clocks,
    }
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        line["cpu_baseline"] = _cpu_baseline(OracleSample(1, 32, P=P, T_=Tw, batch=B, head_rows=16), UNIT,
                                             lambda s: 1.0 / s)
    ctx.close()
    return line


def run_generation(name, args, env):
    import numpy as np
    torch, device, world, rank, pg = env["torch"], env["device"], env["world"], env["rank"], env["pg"]
    from paper_2606_13740_gb300 import Config, Context, Sched

    Lp, gen, kw, what = GENERATIONS[name]
    kw = dict(kw)
    if "spec_allowance" in kw:
        kw["spec_lat"] = tuple(env.get("spec_lat") or (3.37, 3.97, 4.14))
    sched = Sched(**kw)
    cfg = Config(max_batch=1, max_ctx=Lp + gen, max_window=max(Lp, 96 + sched.scr_rows), **SHAPE)
    ctx = Context(cfg)
    prompt = I.uniform_prompt(Lp, cfg.vocab, cfg.mask_id, seed=I.SEED_PROMPT + rank)
    for _ in range(max(1, min(args.warmup, 2))):  # warm-up: the graph of every window shape
        ctx.dllm_generate(sched, prompt, gen)
    ctx.dllm_sync()
    reps = max(1, min(args.steps, 5))
    stats = None
    with Timed(torch, device, ctx.stream, pg) as tm:
        for _ in range(reps):
            _, stats = ctx.dllm_generate(sched, prompt, gen)
    sec = tm.wall / reps
    sec = _max_over_ranks(sec, pg, device)
    value = world * gen / sec
    ctx.dllm_set_profile(1)
    ctx.dllm_generate(sched, prompt, gen)
    prof, psteps = ctx.dllm_get_profile()
    ctx.dllm_set_profile(0)
    ctx.close()

    hbm, bf16, bf16_sus, peak_src = env["peaks"]
    # algorithmic bytes of the generation: every step's weights + prefix K/V, the block appends
    # (layer weights once each) and the prefill (layer weights once)
    steps = stats["steps"]
    P_mid = Lp + gen // 2
    gen_bytes = steps * _step_bytes(P_mid, T) + (stats["blocks"] + 1) * 13.959e9
    ach = gen_bytes / sec / 1e9
    algo = _algorithmic_bytes(T)
    per_layer = algo["oproj"] + algo["gateup"] + algo["down"]
    chain_bytes = (31 * (per_layer + algo["qkv"]) + per_layer + algo["head"]) / 32
    roof = _chain_roofline(prof, psteps, chain_bytes, "GB/s", hbm, peak_src, "hbm",
                           "k_chain (one layer's chained projections; 32-token windows counted)")
    line = {
        "metric": METRIC, "value": value, "unit": GEN_UNIT, "n_gpus": world, "steps": reps,
        "warmup": max(1, min(args.warmup, 2)), "ms_per_step": 1e3 * sec, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": dict(workload=name, model=MODEL, batch=1, prompt=Lp, generated=gen, schedule=kw, what=what,
                       step="one whole generation (prefill, every block and step, appends) through dllm_generate",
                       l2="inputs larger than L2 (15 GB of weights streamed per denoising step)", seeds=SEEDS),
        "denoise_steps": steps, "denoise_steps_per_s": steps / sec, "spec_steps": stats["spec_steps"],
        "spec_step_share": stats["spec_steps"] / max(1, steps), "blocks": stats["blocks"],
        "roofline": roof,
        "gen_roofline": {"bound": "hbm", "algorithmic_bytes_per_generation": gen_bytes, "achieved": ach,
                         "peak": hbm, "unit": "GB/s", "frac": ach / hbm},
        "kernel_ms_per_step": {k: v["ms_total"] / max(1, psteps) for k, v in prof.items()},
        "e2e": {"value": value, "unit": GEN_UNIT, "h2d_bytes_per_step": Lp * 4 + 240,
                "d2h_bytes_per_step": gen * 4 + steps * 32,
                "note": "dllm_generate takes the host prompt and returns host tokens: value is end to end"},
        "clocks": tm.clocks,
    }
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        line["cpu_baseline"] = _cpu_baseline(OracleSample(2, 16, P=P_mid, T_=T), GEN_UNIT,
                                             lambda s: gen / (s * steps * 1.05), min_cpu_s=6.0)
        line["cpu_baseline"]["sample"] += f"; x{steps} steps + 5% for the prefill and appends"
    return line


def run_window_sweep(args, env):
    import numpy as np
    torch, device, world, rank, pg = env["torch"], env["device"], env["world"], env["rank"], env["pg"]
    from paper_2606_13740_gb300 import Config, Context, Sched

    hbm, bf16, bf16_sus, peak_src = env["peaks"]
    rows, clocks = [], []
    for Tw in (32, 64, 96, 128, 192, 256):
        cfg = Config(max_batch=1, max_ctx=LP + Tw, max_window=max(Tw, LP), block_len=Tw, **SHAPE)
        ctx = Context(cfg)
        ctx.dllm_prefill(Sched(steps_per_block=Tw), I.uniform_prompt(LP, cfg.vocab, cfg.mask_id), Tw)
        ctx.dllm_begin_block()  # one block of length Tw: the window, every position masked
        ctx.dllm_set_state(*ctx.dllm_get_state()[:2])

        def step():
            ctx.dllm_rewind_block()
            ctx.dllm_denoise_step(want_out=False)

        for _ in range(3):
            step()
        n = max(3, min(args.steps, 30))
        with Timed(torch, device, ctx.stream, pg) as tm:
            for _ in range(n):
                step()
        ms = tm.ms / n
        clocks.append(tm.clocks)
        b = _step_bytes(LP, Tw)
        rows.append({"T": Tw, "ms_per_step": ms, "steps_per_s": 1e3 / ms, "hbm_frac": b / (ms * 1e-3) / 1e9 / hbm,
                     "tensor_frac": (32 * _layer_flops(Tw) + 2 * Tw * 126464 * 4096) / (ms * 1e-3) / 1e12 / bf16})
        ctx.close()
    r32 = rows[0]
    return {
        "metric": METRIC, "value": r32["steps_per_s"], "unit": UNIT, "n_gpus": world, "steps": n,
        "warmup": 3, "ms_per_step": r32["ms_per_step"], "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": dict(workload=SWEEP, model=MODEL, batch=1, prompt=LP, windows=[r["T"] for r in rows],
                       l2="inputs larger than L2", seeds=SEEDS),
        "rows": rows, "spec_lat": [rows[i]["ms_per_step"] for i in (0, 1, 2)],
        "clocks": clocks[0], "clocks_all": clocks,
    }


def run_ours(args):
    import torch

    world, rank, local, pg = _dist_setup(args)
    torch.cuda.set_device(local)
    device = torch.device("cuda", local)
    env = dict(torch=torch, device=device, world=world, rank=rank, pg=pg, peaks=_peaks())
    names = ALL if args.workload == "all" else [args.workload]
    for name in names:
        if name == WORKLOAD["workload"]:
            line = run_step_b1(args, env)
        elif name == STEP_Q4:
            line = run_step_b1(args, env, q4=True)
        elif name == STEP_B16:
            line = run_step_b16(args, env)
        elif name == SWEEP:
            line = run_window_sweep(args, env)
            env["spec_lat"] = line["spec_lat"]
        else:
            line = run_generation(name, args, env)
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
    ap.add_argument("--workload", choices=ALL + ["all"], default=WORKLOAD["workload"])
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-pdl", action="store_true", help="launch kernels without programmatic dependent launch")
    ap.add_argument("--full-smem", action="store_true", help="one 227 KB projection CTA per SM (no co-residency)")
    args = ap.parse_args(argv)
    if args.impl == "reference":
        return run_reference(args)
    return run_ours(args)


if __name__ == "__main__":
    sys.exit(main())
