"""Seeded synthetic inputs shared by the oracle tests, the GPU tests and the
benchmark.  This module holds none of the decoding arithmetic: it only draws
token ids, mask patterns and scripted confidences from numpy generators.

Workload recipes (the paper's datasets and trained weights are not used; these
stand in for them):
  - prompts: ids uniform over [0, V) without the mask id;
  - batched serving: ids Zipf(1.1)-distributed over ranks 1..V-1 by inverse
    CDF on an fp64 table, rank r -> id r-1 (skipping the mask id);
  - masked window: a seeded choice of which window positions start masked.
"""
from __future__ import annotations

import numpy as np

SEED_WEIGHTS = 0x11ADA8B
SEED_PROMPT = 1
SEED_ZIPF = 2
SEED_KV = 3

TINY = dict(n_layers=2, d_model=256, n_heads=4, head_dim=64, ffn=688, vocab=1024, mask_id=1023,
            rope_base=10000.0, rms_eps=1e-5)
LLADA_8B = dict(n_layers=32, d_model=4096, n_heads=32, head_dim=128, ffn=12288, vocab=126464,
                mask_id=126463, rope_base=500000.0, rms_eps=1e-5)


def uniform_prompt(n: int, vocab: int, mask_id: int, seed: int = SEED_PROMPT, batch: int | None = None):
    """Uniform ids in [0, vocab) excluding mask_id."""
    rng = np.random.default_rng(seed)
    shape = (n,) if batch is None else (batch, n)
    ids = rng.integers(0, vocab - 1, size=shape, dtype=np.int64)
    ids = np.where(ids >= mask_id, ids + 1, ids)
    return ids.astype(np.int32)


def zipf_ids(shape, vocab: int, mask_id: int, s: float = 1.1, seed: int = SEED_ZIPF):
    """Zipf(s) over ranks 1..vocab-1 by inverse CDF; rank r -> id r-1, skipping mask_id."""
    rng = np.random.default_rng(seed)
    ranks = np.arange(1, vocab, dtype=np.float64)
    w = ranks ** (-s)
    cdf = np.cumsum(w)
    cdf /= cdf[-1]
    u = rng.random(size=shape)
    r = np.searchsorted(cdf, u, side="left")  # 0-based rank index
    ids = np.where(r >= mask_id, r + 1, r)
    return np.minimum(ids, vocab - 1).astype(np.int32)


def masked_positions(T: int, n_masked: int, seed: int = SEED_PROMPT + 100):
    """Seeded choice of n_masked of T window positions (sorted)."""
    rng = np.random.default_rng(seed)
    return np.sort(rng.choice(T, size=n_masked, replace=False)).astype(np.int32)


def scripted_confidences(n: int, seed: int, ties: bool = False):
    """Confidence arrays for commit-pass tests; with ties, values repeat."""
    rng = np.random.default_rng(seed)
    if ties:
        return rng.choice(np.array([0.1, 0.25, 0.5, 0.5, 0.75, 0.95], np.float32), size=n)
    return rng.random(n).astype(np.float32)
