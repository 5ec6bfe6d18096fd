"""Pins of the oracle's positional encoding and qk-norm (oracle.position): the reading of
Algorithm 1's undefined positional information P as qk-norm + 2-D RoPE.  The paper prints
no values for P, so these pin the functions to the mathematics they must satisfy."""
import numpy as np
import pytest

import oracle


def test_token_positions_worked_example():
    # two views of 1 camera + 4 register tokens and a 3 x 3 patch grid
    py, px = oracle.token_positions(28, tokens_per_view=14, patch_start=5, grid_w=3)
    view = [(0, 0)] * 5 + [(1, 1), (1, 2), (1, 3), (2, 1), (2, 2), (2, 3), (3, 1), (3, 2), (3, 3)]
    assert list(zip(py.tolist(), px.tolist())) == view + view


def test_rope_preserves_norms_and_separates_axes():
    g = np.random.default_rng(0)
    x = g.standard_normal((50, 64))
    py, px = g.integers(0, 40, 50), g.integers(0, 40, 50)
    y = oracle.rope_2d(x, py, px, 100.0)
    # every rotated plane (channel i, i + 16 inside each half) keeps its length
    for half in (0, 32):
        for i in range(16):
            a = np.hypot(x[:, half + i], x[:, half + i + 16])
            b = np.hypot(y[:, half + i], y[:, half + i + 16])
            np.testing.assert_allclose(a, b, rtol=1e-12)
    # the row position turns only channels [0, 32), the column position only [32, 64)
    y_row = oracle.rope_2d(x, py, np.zeros(50, int), 100.0)
    np.testing.assert_array_equal(y_row[:, 32:], x[:, 32:])
    y_col = oracle.rope_2d(x, np.zeros(50, int), px, 100.0)
    np.testing.assert_array_equal(y_col[:, :32], x[:, :32])
    # position (0, 0) is the identity
    np.testing.assert_allclose(oracle.rope_2d(x, np.zeros(50, int), np.zeros(50, int), 100.0), x)


def test_rope_scores_depend_on_relative_position_only():
    g = np.random.default_rng(1)
    q, k = g.standard_normal((1, 64)), g.standard_normal((1, 64))
    for (qy, qx, ky, kx) in [(1, 2, 5, 7), (3, 3, 3, 3), (10, 1, 2, 30)]:
        ref = float((oracle.rope_2d(q, [qy], [qx], 100.0) @ oracle.rope_2d(k, [ky], [kx], 100.0).T)[0, 0])
        for ty, tx in [(1, 0), (0, 4), (7, 11)]:
            got = float((oracle.rope_2d(q, [qy + ty], [qx + tx], 100.0)
                         @ oracle.rope_2d(k, [ky + ty], [kx + tx], 100.0).T)[0, 0])
            assert got == pytest.approx(ref, rel=1e-10, abs=1e-12)


def test_rope_fastest_and_slowest_planes():
    # plane 0 turns by exactly the position (base^0 = 1), in the direction channel 0 -> 16;
    # plane 15 by position * base^(-15/16)
    x = np.zeros((1, 64))
    x[0, 0] = 1.0
    x[0, 15] = 1.0
    y = oracle.rope_2d(x, [3], [0], 100.0)
    assert y[0, 0] == pytest.approx(np.cos(3.0)) and y[0, 16] == pytest.approx(np.sin(3.0))
    w = 3.0 * 100.0 ** (-15.0 / 16.0)
    assert y[0, 15] == pytest.approx(np.cos(w)) and y[0, 31] == pytest.approx(np.sin(w))


def test_qk_norm_is_layer_norm_over_the_head():
    torch = pytest.importorskip("torch")
    g = np.random.default_rng(2)
    x = 3.0 * g.standard_normal((20, 64)) + 1.5
    gam, bet = 1.0 + 0.1 * g.standard_normal(64), 0.1 * g.standard_normal(64)
    got = oracle.qk_transform(x, (gam, bet), 1e-6, None, None)
    want = torch.nn.functional.layer_norm(torch.from_numpy(x), (64,), torch.from_numpy(gam),
                                          torch.from_numpy(bet), eps=1e-6).numpy()
    np.testing.assert_allclose(got, want, rtol=1e-10, atol=1e-12)
