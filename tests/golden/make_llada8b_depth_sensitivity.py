"""Writes llada8b_depth_sensitivity.json: how much the oracle's own outputs move, layer by
layer, when its input moves by a bf16-sized amount, at the benchmarked configuration.

Calls only the oracle (oracle/) and the seeded input generators (dllm_inputs.py).

Why: the paper's step keeps activations in 16 bits (Sec. 5.1 runs FP16 activations; the GPU
path reads this as bf16 operands with fp32 accumulation).  A randomly initialised 32-layer
model (N(0, 0.02) weights, as the benchmark uses) amplifies any perturbation of its hidden
state: a computation that rounds its operands to bf16 drifts from the fp32 oracle by more
than 1e-2 after a few layers however it is implemented.  The full-depth parity test therefore
bounds the GPU's deviation at layer l by a multiple of this file's amplification A_l times
the bf16 unit roundoff, and keeps 1e-2 wherever that is larger.

How: the oracle runs the benchmark's prefill (512 uniform prompt ids) and one denoising step
(a 32-token window, 24 masked) twice on the same model: as is, and with the embedding rows of
the ids it reads perturbed by one bf16 ulp on a seeded half of their elements.  A_l is the
relative L2 change of the layer-l prefix K (and V) divided by the relative L2 change of those
embedding rows; the same ratio is stored for every window row's logits.

    python tests/golden/make_llada8b_depth_sensitivity.py     # about 15 minutes on 8 cores
"""
import json
import os
import sys
import time

import numpy as np

ROOT = os.path.dirname(os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
sys.path.insert(0, ROOT)

import dllm_inputs as I  # noqa: E402
import oracle as O  # noqa: E402

SHAPE = dict(n_layers=32, d_model=4096, n_heads=32, head_dim=128, ffn=12288, vocab=126464, mask_id=126463,
             rope_base=500000.0)
LP, T, MASKED = 512, 32, 24
OUT = os.path.join(os.path.dirname(os.path.abspath(__file__)), "llada8b_depth_sensitivity.json")


def window_state(tok, st):
    win = np.arange(LP, LP + T)
    tok, st = tok.copy(), st.copy()
    tok[win] = I.uniform_prompt(T, SHAPE["vocab"], SHAPE["mask_id"], seed=7)
    st[win] = O.COMMITTED
    m = win[I.masked_positions(T, MASKED)]
    tok[m], st[m] = SHAPE["mask_id"], O.MASKED
    return tok, st


def run(model, prompt):
    sess = O.Session(model, O.OracleSched(steps_per_block=MASKED), prompt, T)
    sess.prefill()
    sess.begin_block()
    tok, st, _ = sess.state()
    w_tok, w_st = window_state(tok, st)
    sess.set_state(w_tok, w_st)
    sess.step(keep_logits=True)
    logits = sess.decisions(logits=True)["logits"].copy()
    k = [sess.prefix_kv(l, 0) for l in range(SHAPE["n_layers"])]
    v = [sess.prefix_kv(l, 1) for l in range(SHAPE["n_layers"])]
    return w_tok, k, v, logits


def main():
    O.build()
    t0 = time.time()
    prompt = I.uniform_prompt(LP, SHAPE["vocab"], SHAPE["mask_id"], seed=I.SEED_PROMPT)
    model = O.Model(O.OracleConfig(**SHAPE))
    w_tok, k0, v0, lg0 = run(model, prompt)
    print(f"clean run {time.time() - t0:.0f} s", flush=True)
    # one bf16 ulp on a seeded half of the elements of every embedding row the two runs read
    emb = model.weight(-1, O.T_EMBED)
    ids = np.unique(np.concatenate([prompt, w_tok[LP:]]))
    before = emb[ids].copy()
    flip = np.random.default_rng(11).random(before.shape) < 0.5
    emb[ids] = before ^ flip.astype(np.uint16)
    after = emb[ids].copy()
    f0 = (before.astype(np.uint32) << 16).view(np.float32)
    f1 = (after.astype(np.uint32) << 16).view(np.float32)
    d_in = float(np.linalg.norm(f1 - f0) / np.linalg.norm(f0))
    _, k1, v1, lg1 = run(model, prompt)
    print(f"both runs {time.time() - t0:.0f} s, input change {d_in:.3e}", flush=True)

    def rel(a, b):
        return float(np.linalg.norm(a - b) / np.linalg.norm(a))

    out = {
        "what": "amplification A = (relative L2 change of an output) / (relative L2 change of the input "
                "embedding rows) of the oracle at the benchmarked configuration: LLaDA-8B shape, 32 layers, "
                "seed 0x11ADA8B weights, 512-token uniform prompt (seed 1), one step on a 32-token window with "
                "24 masked; written by tests/golden/make_llada8b_depth_sensitivity.py from the oracle only",
        "citation": "Sec. 5.1 (16-bit activations on the NPU; read as bf16 operands with fp32 accumulation)",
        "u_bf16": 2.0 ** -8,
        "delta_in": d_in,
        "A_K": [rel(k0[l], k1[l]) / d_in for l in range(SHAPE["n_layers"])],
        "A_V": [rel(v0[l], v1[l]) / d_in for l in range(SHAPE["n_layers"])],
        "A_logits_rows": [rel(lg0[r], lg1[r]) / d_in for r in range(T)],
    }
    with open(OUT, "w") as f:
        json.dump(out, f, indent=1)
    print(json.dumps({k: (v if not isinstance(v, list) else [round(x, 3) for x in v[:4]] + ["..."])
                      for k, v in out.items()}))


if __name__ == "__main__":
    main()
