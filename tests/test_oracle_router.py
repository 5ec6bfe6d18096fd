"""Pins of the oracle's router (§4.1) and routing rule (§4.2) against closed forms."""
import json
import math
import os

import numpy as np
import pytest

import oracle
from oracle import MODE_FULL, MODE_MEAN, MODE_SURROGATE

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def test_pooling_worked_example_closed_form():
    # d = L = 2, W = I, U = 0 (sigma(0) = 1/2), w = (4, 0): the pooling logit of
    # token i is 4 * 1/2 * tanh(q_i0) = 2 tanh(q_i0).  Choosing q_i0 =
    # atanh(t_i / 2) with t = (0, ln 2, ln 3) makes the logits (0, ln 2, ln 3),
    # so alpha = (1, 2, 3) / 6 exactly.
    t = np.array([0.0, math.log(2.0), math.log(3.0)])
    q0 = np.arctanh(t / 2.0)
    q1 = np.array([5.0, -1.0, 2.0])
    Q = np.stack([q0, q1], axis=1)
    W, U, w = np.eye(2), np.zeros((2, 2)), np.array([4.0, 0.0])
    alpha, q_pool = oracle.attention_pool(Q, W, U, w)
    np.testing.assert_allclose(alpha, [1 / 6, 2 / 6, 3 / 6], rtol=1e-14)
    np.testing.assert_allclose(q_pool[1], (5.0 - 2.0 + 6.0) / 6.0, rtol=1e-14)
    np.testing.assert_allclose(q_pool[0], (2 * q0[1] + 3 * q0[2]) / 6.0, rtol=1e-14)
    # Swapping the roles of W and U gives tanh(0) = 0 logits, hence uniform alpha:
    # a transposed or swapped operand would fail the assertion above.
    alpha_sw, _ = oracle.attention_pool(Q, U, W, w)
    np.testing.assert_allclose(alpha_sw, [1 / 3] * 3, rtol=1e-14)


def test_pooling_bias_terms():
    # With W = 0 and bias bW = atanh(0.5) on the first channel, tanh(W q + bW) = 0.5;
    # with U = 0 and bU = 0, the gate is 1/2: every logit equals w0 * 0.25.
    Q = np.random.default_rng(0).standard_normal((9, 2))
    e = oracle.pooling_logits(Q, np.zeros((2, 2)), np.zeros((2, 2)), np.array([8.0, 1.0]),
                              bW=np.array([np.arctanh(0.5), 0.0]), bU=np.zeros(2))
    np.testing.assert_allclose(e, 2.0, rtol=1e-14)


def test_identical_queries_pool_to_that_query():
    g = np.random.default_rng(3)
    q = g.standard_normal(64)
    Q = np.tile(q, (50, 1))
    W, U, w = g.standard_normal((64, 64)), g.standard_normal((64, 64)), g.standard_normal(64)
    _, q_pool = oracle.attention_pool(Q, W, U, w)
    np.testing.assert_allclose(q_pool, q, rtol=1e-13, atol=1e-14)


def test_zero_score_vector_gives_mean_query():
    g = np.random.default_rng(4)
    Q = g.standard_normal((77, 64))
    alpha, q_pool = oracle.attention_pool(Q, g.standard_normal((64, 64)), g.standard_normal((64, 64)),
                                          np.zeros(64))
    np.testing.assert_allclose(alpha, 1 / 77, rtol=1e-14)
    np.testing.assert_allclose(q_pool, Q.mean(axis=0), rtol=1e-12, atol=1e-14)


def test_alpha_and_r_sum_to_one():
    g = np.random.default_rng(5)
    Q, K = g.standard_normal((300, 64)), g.standard_normal((300, 64))
    alpha, q_pool = oracle.attention_pool(Q, g.standard_normal((64, 64)), g.standard_normal((64, 64)),
                                          g.standard_normal(64) * 5)
    r = oracle.routing_vector(q_pool * 3, K, 1 / 8)
    assert abs(alpha.sum() - 1) < 1e-14 and abs(r.sum() - 1) < 1e-14
    assert np.all(alpha >= 0) and np.all(r >= 0)
    assert oracle.saliency(r) == r.max()


def test_identical_keys_give_saliency_one_over_n():
    for N in (1, 7, 100, 1044):
        K = np.tile(np.random.default_rng(N).standard_normal(64), (N, 1))
        r = oracle.routing_vector(np.random.default_rng(0).standard_normal(64), K, 0.125)
        np.testing.assert_allclose(oracle.saliency(r), 1.0 / N, rtol=1e-14)


@pytest.mark.parametrize("N,gap", [(2, 0.0), (10, 1.0), (1000, 5.0), (5000, 12.0)])
def test_single_dominant_key_closed_form(N, gap):
    # Keys: e_1 for key 0, zero for the rest; q_pool = gap * sqrt(d) / beta * e_1,
    # so the routing logits are (gap, 0, ..., 0) and s = 1 / (1 + (N-1) e^-gap).
    d, beta = 64, 1.0
    K = np.zeros((N, d))
    K[0, 0] = 1.0
    q = np.zeros(d)
    q[0] = gap * math.sqrt(d) / beta
    r = oracle.routing_vector(q, K, beta / math.sqrt(d))
    np.testing.assert_allclose(oracle.saliency(r), 1.0 / (1.0 + (N - 1) * math.exp(-gap)), rtol=1e-13)


def test_saliency_monotone_in_temperature():
    g = np.random.default_rng(6)
    K, q = g.standard_normal((2000, 64)), g.standard_normal(64) * 0.3
    s = [oracle.saliency(oracle.routing_vector(q, K, b / 8)) for b in np.geomspace(0.01, 1e4, 60)]
    assert all(b >= a - 1e-15 for a, b in zip(s, s[1:]))
    assert s[0] < 2.0 / 2000 and s[-1] > 0.99


def test_select_mode_cases_and_ties():
    f32 = np.float32
    lo, hi = f32(0.01), f32(0.2)
    assert oracle.select_mode(hi) == MODE_FULL                    # s = tau_high -> full
    assert oracle.select_mode(lo) == MODE_MEAN                    # s = tau_low -> mean
    assert oracle.select_mode(np.nextafter(hi, f32(0))) == MODE_SURROGATE
    assert oracle.select_mode(np.nextafter(lo, f32(1))) == MODE_SURROGATE
    assert oracle.select_mode(np.nextafter(lo, f32(0))) == MODE_MEAN
    assert oracle.select_mode(1.0) == MODE_FULL
    assert oracle.select_mode(0.0) == MODE_MEAN
    assert oracle.select_mode(0.05) == MODE_SURROGATE
    assert oracle.select_mode(float("nan")) == MODE_FULL
    # Two-way router (tau_low = tau_high): every head is full or mean.
    for s in (0.0, 0.05, 0.1, 0.2, 0.7):
        assert oracle.select_mode(s, f32(0.1), f32(0.1)) in (MODE_FULL, MODE_MEAN)
    assert oracle.select_mode(0.1, f32(0.1), f32(0.1)) == MODE_FULL
    # The decision is taken in float32: a float64 saliency a hair below tau_high
    # that rounds to tau_high in float32 is full.
    assert oracle.select_mode(0.2 - 1e-12) == MODE_FULL


def test_thresholds_match_paper_constants():
    c = json.load(open(os.path.join(GOLDEN, "paper_constants.json")))
    from oracle.layer import TAU_HIGH, TAU_LOW
    assert TAU_LOW == np.float32(c["tau_low"]["value"])
    assert TAU_HIGH == np.float32(c["tau_high"]["value"])


def test_bin_heads_is_a_stable_partition():
    g = np.random.default_rng(7)
    for trial in range(50):
        H = int(g.integers(1, 33))
        N = int(g.integers(1, 5000))
        modes = g.integers(0, 3, H).astype(np.int32)
        ids, off, work = oracle.bin_heads(modes, N)
        assert sorted(ids.tolist()) == list(range(H))
        assert off[0] == 0 and off[-1] == H and np.all(np.diff(off) >= 0)
        for m in range(3):
            seg = ids[off[m]:off[m + 1]]
            assert np.all(modes[seg] == m) and np.all(np.diff(seg) > 0)
        n_tiles = -(-N // 128)
        assert len(work) == (modes == MODE_FULL).sum() * n_tiles
        # Brute force: every (full head, tile) pair exactly once, head-major.
        expect = [(h, t) for h in range(H) if modes[h] == MODE_FULL for t in range(n_tiles)]
        assert [tuple(x) for x in work.tolist()] == expect


def test_mean_query_pooling_ablation():
    """§5 component ablation: Q-Pooling replaced by mean pooling, independent of the weights."""
    g = np.random.default_rng(41)
    N, d = 37, 64
    Q = g.standard_normal((N, d))
    for _ in range(2):
        W, U, w = g.standard_normal((64, d)), g.standard_normal((64, d)), g.standard_normal(64)
        alpha, qp = oracle.attention_pool(Q, W, U, w, mean_pool=True)
        np.testing.assert_allclose(alpha, np.full(N, 1.0 / N), rtol=1e-15)
        np.testing.assert_allclose(qp, Q.mean(0), rtol=1e-12, atol=1e-15)


def test_two_branch_routing_has_no_surrogate_band():
    """§5 compute-mode ablation "mean + full only": tau_low == tau_high leaves no band."""
    t = np.float32(0.05)
    for s in np.float32([0.0, 0.01, 0.049, 0.05, 0.0500001, 0.3, 1.0]):
        m = oracle.select_mode(s, t, t)
        assert m == (oracle.MODE_FULL if s >= t else oracle.MODE_MEAN)
