"""Pins of the oracle's counter-based weight generator.

The generator is not from the paper (it used trained weights); it is the
seeded stand-in.  Each side implements it from the SplitMix64 definition, so
these pins fix the definition itself: published SplitMix64 outputs, the
Irwin-Hall(4) distribution's moments, and bf16 round-to-nearest-even against
torch's own conversion.
"""
import os

import numpy as np
import pytest
import torch

import oracle as O

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "splitmix64_state0.txt")


def test_splitmix64_published_outputs(oracle_lib):
    rows = [ln.split() for ln in open(GOLDEN) if ln.strip() and not ln.startswith("#")]
    L = O.lib()
    for n, val in rows:
        assert L.orc_splitmix_at(0, int(n)) == int(val, 16)


def test_irwin_hall_moments(oracle_lib):
    x = O.gen_f32(0x11ADA8B, 16, 0, 1 << 20, 1.0).astype(np.float64)
    n = x.size
    assert abs(x.mean()) < 5.0 / np.sqrt(n)
    assert abs(x.var() - 1.0) < 0.01
    # Irwin-Hall of order 4 (centred): support +-2*sqrt(3), excess kurtosis -6/(5*4)
    assert np.abs(x).max() <= 2 * np.sqrt(3) + 1e-6
    kurt = ((x - x.mean()) ** 4).mean() / x.var() ** 2 - 3.0
    assert abs(kurt - (-0.3)) < 0.02


def test_sigma_scaling_and_independence(oracle_lib):
    a = O.gen_f32(7, 16, 0, 4096, 1.0)
    b = O.gen_f32(7, 16, 0, 4096, 0.02)
    assert np.allclose(b, (a.astype(np.float64) * 0.02).astype(np.float32), rtol=1e-6, atol=0)
    c = O.gen_f32(7, 17, 0, 4096, 1.0)
    assert abs(np.corrcoef(a, c)[0, 1]) < 0.06
    # counter-based: any slice equals the same slice of a longer draw
    d = O.gen_f32(7, 16, 1000, 96, 1.0)
    assert np.array_equal(d, a[1000:1096])


def test_bf16_round_to_nearest_even_matches_torch(oracle_lib):
    rng = np.random.default_rng(0)
    x = np.concatenate([rng.standard_normal(5000).astype(np.float32) * 0.02,
                        np.array([1.0, -0.0, 1.00390625, 1.01171875, 3.0e38, 1e-40], np.float32)])
    ours = O.f32_to_bf16_bits(x)
    ref = torch.from_numpy(x).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    assert np.array_equal(ours, ref)


def test_gen_bf16_is_rounded_gen_f32(oracle_lib):
    f = O.gen_f32(3, 20, 0, 10000, 0.02)
    h = O.gen_bf16(3, 20, 0, 10000, 0.02)
    ref = torch.from_numpy(f).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    assert np.array_equal(h, ref)


@pytest.mark.parametrize("i", [0, 1, 12345, 2 ** 33 + 5])
def test_element_definition_in_python_floats(oracle_lib, i):
    """Each element is exact integer ops then correctly rounded double ops."""
    L = O.lib()
    seed, tid, sigma = 0x11ADA8B, 17, 0.02
    key = L.orc_splitmix_at(seed, tid)
    s = sum(L.orc_splitmix_at(key, 4 * i + j) >> 32 for j in range(4))
    z = (float(s) - 2.0 ** 33) * float.fromhex("0x1.bb67ae8584caap-32")
    want = np.float32(z * sigma)
    got = O.gen_f32(seed, tid, i, 1, sigma)[0]
    assert got == want
