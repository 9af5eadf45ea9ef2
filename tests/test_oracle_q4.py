"""Pins of the oracle's 4-bit block-quantised weights (the Q4_0 weights the paper runs, Sec. 5.1):
32 consecutive weights of a row share a scale d; a weight is a 4-bit code q and stands for
d * (q - 8), which the arithmetic uses rounded once to bf16.

- A hand-worked block: scale 1 + 1/128, every code, the bf16 values worked out by hand.
- With power-of-two scales the format is exact (no rounding): d * (q - 8) itself.
- Otherwise the rounding stays within half a bf16 ulp of d * (q - 8): 2^-8 relative (8 significant
  bits).
- The synthetic draws: codes uniform over 0..15, scales (1 + m/128) 2^-8 with m < 32 (weights of
  standard deviation 0.02, like the bf16 draws), one scale per block of 32, and a model in the
  format holds exactly those dequantised weights.
"""
from fractions import Fraction

import numpy as np
import pytest

import dllm_inputs as I
import oracle as O


@pytest.fixture(scope="module")
def lib(oracle_lib):
    return oracle_lib


def _bf16_value(bits):
    """Exact value of bf16 bits as a Fraction (sign, 8-bit exponent, 7-bit mantissa)."""
    sign = -1 if bits & 0x8000 else 1
    e = (bits >> 7) & 0xFF
    m = bits & 0x7F
    assert 0 < e < 255
    return sign * Fraction(128 + m, 128) * Fraction(2) ** (e - 127)


def _ulp(x):
    """Spacing of bf16 values at |x| (8 significant bits)."""
    x = abs(x)
    e = 0
    while Fraction(2) ** (e + 1) <= x:
        e += 1
    while Fraction(2) ** e > x:
        e -= 1
    return Fraction(2) ** (e - 7)


def test_hand_worked_block(lib):
    s = 0x3F81  # 1 + 1/128
    # (q - 8) * (1 + 1/128) rounded to 8 significant bits, ties to even, by hand:
    expect = {
        0: 0xC101,   # -8.0625 = -1.0000001b x 2^3: exact
        1: 0xC0E2,   # -7.0546875 = -1.11000011|1b x 2^2 -> -1.1100010b x 2^2 = -7.0625
        5: 0xC042,   # -3.0234375 = -1.1000001|1b x 2 (a tie) -> even: -1.1000010b x 2 = -3.03125
        7: 0xBF81,   # -1.0078125: exact
        8: 0x0000,   # 0
        9: 0x3F81,   # 1.0078125
        10: 0x4001,  # 2.015625 = 1.0000001b x 2: exact
        11: 0x4042,  # 3.0234375 -> 3.03125 (tie to even)
        15: 0x40E2,  # 7.0546875 -> 7.0625
    }
    for q, bits in expect.items():
        got = O.q4_dequant(q, s)
        assert got == bits, (q, hex(got), hex(bits))
    assert _bf16_value(O.q4_dequant(15, s)) == Fraction(113, 16)


def test_power_of_two_scales_are_exact(lib):
    for e in range(-12, 4):
        sbits = (127 + e) << 7  # 2^e
        for q in range(16):
            got = O.q4_dequant(q, sbits)
            want = Fraction(q - 8) * Fraction(2) ** e
            assert (got == 0 and want == 0) or _bf16_value(got) == want


def test_rounding_within_half_an_ulp(lib):
    rng = np.random.default_rng(0)
    for sbits in list(rng.integers(0x3B80, 0x3C00, 64)) + list(rng.integers(0x3000, 0x4400, 64)):
        d = _bf16_value(int(sbits))
        for q in range(16):
            exact = d * (q - 8)
            got = O.q4_dequant(q, int(sbits))
            if exact == 0:
                assert got == 0
                continue
            err = abs(_bf16_value(got) - exact)
            assert err <= abs(exact) * Fraction(1, 256), (hex(int(sbits)), q)
            assert err <= Fraction(1, 2) * _ulp(exact)


def test_synthetic_draws(lib):
    seed, tid, rows, cols = I.SEED_WEIGHTS, 16 + 8 * 3 + 4, 64, 200
    codes = np.array([[O.q4_code(seed, tid, cols, r, c) for c in range(cols)] for r in range(rows)])
    hist = np.bincount(codes.ravel(), minlength=16)
    n = codes.size
    chi2 = float(((hist - n / 16) ** 2 / (n / 16)).sum())
    assert chi2 < 45.0  # 15 degrees of freedom: p < 1e-4 above this
    nblk = (cols + 31) // 32
    scales = np.array([[O.q4_scale(seed, tid, cols, r, b) for b in range(nblk)] for r in range(rows)])
    assert scales.min() >= 0x3B80 and scales.max() <= 0x3B9F  # (1 + m/128) 2^-8, m < 32
    assert len(np.unique(scales)) == 32
    # the weights' spread is that of the bf16 draws, N(0, 0.02)
    wf = (O.gen_q4(seed, tid, 512, 256).astype(np.uint32) << 16).view(np.float32)
    assert abs(float(wf.std()) - 0.02) < 0.001
    w = O.gen_q4(seed, tid, rows, cols)
    for r in (0, 17, 63):
        for c in (0, 31, 32, 199):
            assert w[r, c] == O.q4_dequant(codes[r, c], scales[r, c // 32])
    # distinct tensors and distinct streams for codes and scales
    assert not np.array_equal(O.gen_q4(seed, tid + 1, rows, cols), w)


def test_model_in_the_format_holds_the_dequantised_weights(lib):
    cfg = O.OracleConfig(weight_bits=4)
    model = O.Model(cfg)
    for layer in range(cfg.n_layers):
        for which in range(7):
            wt = model.weight(layer, which)
            assert np.array_equal(wt, O.gen_q4(cfg.weight_seed, 16 + 8 * layer + which, *wt.shape)), (layer, which)
    head = model.weight(-1, O.T_HEAD)
    assert np.array_equal(head, O.gen_q4(cfg.weight_seed, O.T_HEAD, cfg.vocab, cfg.d_model))
    emb = model.weight(-1, O.T_EMBED)  # the embedding stays bf16 N(0, 0.02)
    assert np.array_equal(emb[3], O.gen_bf16(cfg.weight_seed, O.T_EMBED, 3 * cfg.d_model, cfg.d_model, 0.02))
    # the forward is the bf16 path's forward on those weights
    zero = O.Model(O.OracleConfig(), zero=True)
    for layer in range(cfg.n_layers):
        for which in range(7):
            zero.weight(layer, which)[:] = model.weight(layer, which)
    zero.weight(-1, O.T_HEAD)[:] = head
    zero.weight(-1, O.T_EMBED)[:] = emb
    tok = I.uniform_prompt(16, 1024, 1023, seed=2)
    pos = np.arange(16, dtype=np.int32)
    assert np.array_equal(O.forward(model, tok, pos)["logits"], O.forward(zero, tok, pos)["logits"])
