"""Pins of the oracle's scalar building blocks against independent definitions."""
import numpy as np
import pytest
import scipy.special
import scipy.stats
import torch

import oracle
from oracle.numerics import BF16_MAX


def test_round_bf16_matches_torch_on_float32_values():
    g = np.random.default_rng(0)
    x = np.concatenate([g.standard_normal(20000) * 10.0 ** g.integers(-30, 30, 20000),
                        g.standard_normal(1000)]).astype(np.float32)
    ours = oracle.round_bf16(x.astype(np.float64))
    ref = torch.from_numpy(x).to(torch.bfloat16).to(torch.float64).numpy()
    np.testing.assert_array_equal(ours, ref)


def test_round_bf16_ties_to_even_and_ranges():
    # 1 + 2^-8 lies halfway between 1 and 1 + 2^-7: ties go to the even significand (1).
    assert oracle.round_bf16(1.0 + 2.0 ** -8) == 1.0
    # 1 + 3*2^-8 lies halfway between 1 + 2^-7 (odd) and 1 + 2^-6 (even).
    assert oracle.round_bf16(1.0 + 3 * 2.0 ** -8) == 1.0 + 2.0 ** -6
    assert oracle.round_bf16(-(1.0 + 3 * 2.0 ** -8)) == -(1.0 + 2.0 ** -6)
    # Just above the halfway point rounds up.
    assert oracle.round_bf16(1.0 + 2.0 ** -8 + 2.0 ** -30) == 1.0 + 2.0 ** -7
    # Subnormal spacing 2^-133; overflow to inf past the largest finite value.
    assert oracle.round_bf16(2.0 ** -133 * 1.4) == 2.0 ** -133
    assert oracle.round_bf16(BF16_MAX) == BF16_MAX
    assert np.isinf(oracle.round_bf16(2.0 ** 128))
    assert oracle.round_bf16(0.0) == 0.0


def test_bf16_decode_roundtrip():
    u = np.arange(0, 65536, 7, dtype=np.uint32).astype(np.uint16)
    v = oracle.bf16_bits_to_f64(u)
    finite = np.isfinite(v)
    ref = torch.from_numpy(u.view(np.int16)).view(torch.bfloat16).to(torch.float64).numpy()
    np.testing.assert_array_equal(v[finite], ref[finite])


def test_gelu_is_x_times_normal_cdf():
    x = np.linspace(-8, 8, 2001)
    np.testing.assert_allclose(oracle.gelu(x), x * scipy.stats.norm.cdf(x), rtol=1e-13, atol=1e-15)
    t = torch.from_numpy(x)
    np.testing.assert_allclose(oracle.gelu(x), torch.nn.functional.gelu(t).numpy(), rtol=1e-13, atol=1e-15)


def test_sigmoid_matches_expit():
    x = np.linspace(-40, 40, 801)
    np.testing.assert_allclose(oracle.sigmoid(x), scipy.special.expit(x), rtol=1e-14, atol=0)
    assert oracle.sigmoid(0.0) == 0.5


def test_softmax_sums_to_one_and_matches_scipy():
    g = np.random.default_rng(1)
    v = g.standard_normal((7, 333)) * 30
    p = oracle.softmax(v, axis=1)
    np.testing.assert_allclose(p.sum(axis=1), 1.0, rtol=0, atol=1e-14)
    np.testing.assert_allclose(p, scipy.special.softmax(v, axis=1), rtol=1e-12, atol=1e-300)
    # Shift invariance (a definition-level property).
    np.testing.assert_allclose(oracle.softmax(v + 123.0, axis=1), p, rtol=1e-12)


def test_layer_norm_matches_torch():
    g = np.random.default_rng(2)
    x = g.standard_normal((5, 1024)) * 3 + 1
    gam, bet = g.standard_normal(1024), g.standard_normal(1024)
    ref = torch.nn.functional.layer_norm(torch.from_numpy(x), (1024,), torch.from_numpy(gam),
                                         torch.from_numpy(bet), eps=1e-6).numpy()
    np.testing.assert_allclose(oracle.layer_norm(x, gam, bet, 1e-6), ref, rtol=1e-12, atol=1e-12)
