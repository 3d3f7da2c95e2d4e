"""Pins of the seeded input generator (synth) and the oracle's C regenerator."""
import os

import numpy as np
import pytest
import torch

import synth
from oracle import cgen

GOLD = os.path.join(os.path.dirname(__file__), "golden")


def _golden_ints(name):
    with open(os.path.join(GOLD, name)) as f:
        return [int(line) for line in f if line.strip() and not line.startswith("#")]


def test_splitmix64_published_vector():
    assert synth.splitmix64_sequence(1234567, 5) == _golden_ints("splitmix64_seed1234567.txt")


def test_numpy_draws_equal_python_ints():
    key = synth.stream_key(9, 4, 3, 2)
    idx = np.array([0, 1, 2, 77, 123456789, 2**40 + 5], dtype=np.uint64)
    got = synth.draws(key, idx)
    want = [synth.mix64_int(key + (int(n) + 1) * synth.GOLDEN) for n in idx]
    assert [int(v) for v in got] == want


def test_normal_is_lane_sum():
    # z = (sum of the twelve 16-bit lanes of draws 3i..3i+2 - 393210) / 65536
    key = synth.stream_key(1, 2, 3, 4)
    for i in (0, 5, 999):
        s = 0
        for k in range(3):
            d = synth.mix64_int(key + (3 * i + k + 1) * synth.GOLDEN)
            s += sum((d >> (16 * j)) & 0xFFFF for j in range(4))
        z = synth.normal_at(key, np.array([i], dtype=np.uint64))[0]
        assert z == np.float32((s - 393210) / 65536.0)


def test_normal_moments_and_support():
    z = synth.normal_range(synth.stream_key(0, synth.T_WQ, 0, 0), 0, 1_000_000).astype(np.float64)
    assert abs(z.mean()) < 5e-3
    assert abs(z.var() - 1.0) < 5e-3
    assert z.min() >= -6.0 and z.max() <= 6.0
    # Irwin-Hall(12) kurtosis is 3 - 1.2/12 = 2.9 (slightly platykurtic)
    kurt = np.mean(z ** 4) / z.var() ** 2
    assert abs(kurt - 2.9) < 0.05


def test_bf16_rounding_matches_torch():
    rng = np.random.default_rng(0)
    x = rng.standard_normal(100_000).astype(np.float32) * np.float32(3.0)
    # include exact ties between two bf16 values (low 16 bits == 0x8000)
    ties = (rng.integers(0, 2**16, 1000).astype(np.uint32) << 16 | 0x8000).view(np.float32)
    ties = ties[np.isfinite(ties)]
    x = np.concatenate([x, ties])
    want = torch.from_numpy(x).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    assert np.array_equal(synth.bf16_bits(x), want)


def test_c_regenerator_matches_numpy():
    key = synth.stream_key(3, synth.T_WGATE, 5, 0)
    a = cgen.normal(key, 12345, 20000, synth.WEIGHT_SIGMA)
    b = synth.scaled(synth.normal_range(key, 12345, 20000), synth.WEIGHT_SIGMA)
    assert np.array_equal(a.view(np.uint32), b.view(np.uint32))
    assert cgen.stream_key(3, 5, 7, 9) == synth.stream_key(3, 5, 7, 9)


def test_turn_assignment_ranges():
    t = synth.turn_assignment(5, 2000, 5, 0.1, 256, 2048)
    plans = np.array([p for p, _ in t])
    lens = np.array([n for _, n in t])
    assert plans.min() >= 0 and plans.max() <= 5
    assert 0.07 < np.mean(plans == 5) < 0.13
    assert lens.min() >= 256 and lens.max() <= 2048


@pytest.mark.parametrize("sigma", [1.0, 0.02])
def test_scaled_is_single_multiply(sigma):
    z = synth.normal_range(synth.stream_key(2, 1, 0, 0), 0, 1000)
    got = synth.scaled(z, sigma)
    want = (z.astype(np.float64) * np.float64(np.float32(sigma))).astype(np.float32)
    assert np.array_equal(got, want)  # a product of two floats rounds once to the nearest float
