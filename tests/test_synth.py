"""Pins for the seeded input generator shared by the oracle and the CUDA path."""
import os

import numpy as np

import synth

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "philox4x32_10_kat.txt")


def test_philox_known_answers():
    rows = [l.split() for l in open(GOLDEN) if l.strip() and not l.startswith("#")]
    assert len(rows) == 3
    for r in rows:
        v = [int(x, 16) for x in r]
        out = synth.philox4x32_10(v[0:4], v[4:6])
        assert [int(x) for x in out] == v[6:10]


def test_weight_moments_and_support():
    sigma = 0.02
    w = synth.weights_f32(0, 16, 0, 1 << 20, sigma).astype(np.float64)
    n = w.size
    # Irwin-Hall(4) centred: mean 0, variance sigma^2, support +-2*sqrt(3)*sigma
    assert abs(w.mean()) < 5 * sigma / np.sqrt(n)
    assert abs(w.var() / sigma**2 - 1.0) < 5 * np.sqrt(2.0 / n) * 1.2
    assert np.abs(w).max() <= 2 * np.sqrt(3) * sigma * (1 + 1e-6)
    # excess kurtosis of a sum of 4 uniforms is -6/(5*4) = -0.3
    kurt = ((w - w.mean()) ** 4).mean() / w.var() ** 2 - 3.0
    assert abs(kurt + 0.3) < 0.02
    # symmetric: odd moment near zero
    assert abs(((w / sigma) ** 3).mean()) < 0.02


def test_streams_differ_by_tensor_and_seed():
    a = synth.weights_f32(0, 16, 0, 64, 1.0)
    b = synth.weights_f32(0, 17, 0, 64, 1.0)
    c = synth.weights_f32(1, 16, 0, 64, 1.0)
    assert not np.array_equal(a, b) and not np.array_equal(a, c)
    # counter addressing: a window equals the same elements of a longer fill
    d = synth.weights_f32(0, 16, 32, 32, 1.0)
    assert np.array_equal(a[32:], d)


def test_bf16_round_to_nearest_even():
    # bf16 rounding of fp32 values that sit exactly between two bf16 values
    # rounds to the even neighbour; above / below the midpoint rounds normally.
    f = np.array([0x3F808000, 0x3F818000, 0x3F808001, 0x3F807FFF], dtype=np.uint32).view(np.float32)
    sig = 1.0
    # use the fill path's rounding by checking bf16 fill == round(f32 fill)
    w32 = synth.weights_f32(3, 20, 0, 4096, sig)
    b16 = synth.weights_bf16_bits(3, 20, 0, 4096, sig)
    u = w32.view(np.uint32)
    expect = ((u + 0x7FFF + ((u >> 16) & 1)) >> 16).astype(np.uint16)
    assert np.array_equal(expect, b16)
    # the midpoint cases by hand
    hand = {0x3F808000: 0x3F80, 0x3F818000: 0x3F82, 0x3F808001: 0x3F81, 0x3F807FFF: 0x3F80}
    for fv, want in zip(f.view(np.uint32), hand.values()):
        got = (int(fv) + 0x7FFF + ((int(fv) >> 16) & 1)) >> 16
        assert got == want


def test_prompt_ids_uniform_in_range():
    ids = synth.prompt_ids(200000, 1000)
    assert ids.min() >= 0 and ids.max() < 1000
    counts = np.bincount(ids, minlength=1000)
    chi2 = ((counts - 200.0) ** 2 / 200.0).sum()
    assert chi2 < 1000 + 6 * np.sqrt(2 * 1000)


def test_qnet_params_bounds():
    p = synth.qnet_hidden_params(3, 64)
    assert p.size == 64 * 3 + 64 + 2 * 64 + 2
    w1 = p[:192]
    w2 = p[256:256 + 128]
    assert np.abs(w1).max() < 1 / np.sqrt(3) and np.abs(w2).max() < 1 / np.sqrt(64)
    assert np.abs(w1).max() > 0.5 / np.sqrt(3)
