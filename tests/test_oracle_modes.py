"""Pins of the oracle's computation modes: full (Algorithm 1), surrogate (§4.3), mean."""
import math

import numpy as np
import scipy.special
import scipy.stats
import torch

import oracle


def test_full_attention_matches_library_sdpa():
    g = np.random.default_rng(0)
    for N, d in ((1, 64), (5, 4), (300, 64), (257, 16)):
        Q, K, V = (g.standard_normal((N, d)) * 2 for _ in range(3))
        ref = torch.nn.functional.scaled_dot_product_attention(
            *(torch.from_numpy(a)[None, None] for a in (Q, K, V)))[0, 0].numpy()
        np.testing.assert_allclose(oracle.full_attention(Q, K, V), ref, rtol=1e-11, atol=1e-12)


def test_full_attention_brute_force_tiny():
    # Element-by-element definition on a 3-token, 2-channel problem.
    Q = np.array([[1.0, 0.0], [0.0, 2.0], [1.0, -1.0]])
    K = np.array([[0.5, 1.0], [-1.0, 0.0], [2.0, 1.0]])
    V = np.array([[1.0, 2.0], [3.0, -1.0], [0.0, 4.0]])
    out = oracle.full_attention(Q, K, V)
    for i in range(3):
        logits = [sum(Q[i, c] * K[j, c] for c in range(2)) / math.sqrt(2) for j in range(3)]
        w = [math.exp(x) for x in logits]
        z = sum(w)
        for c in range(2):
            assert abs(out[i, c] - sum(w[j] / z * V[j, c] for j in range(3))) < 1e-14


def test_full_attention_special_cases():
    g = np.random.default_rng(1)
    N, d = 200, 64
    Q, V = g.standard_normal((N, d)), g.standard_normal((N, d))
    # Identical keys: uniform weights, every row is the mean of V.
    K = np.tile(g.standard_normal(d), (N, 1))
    np.testing.assert_allclose(oracle.full_attention(Q, K, V), np.tile(V.mean(0), (N, 1)), rtol=1e-12, atol=1e-13)
    # Constant V: output equals V.
    Vc = np.tile(g.standard_normal(d), (N, 1))
    np.testing.assert_allclose(oracle.full_attention(Q, g.standard_normal((N, d)), Vc), Vc, rtol=1e-12)
    # V = identity (d = N): the output is the attention matrix; rows sum to one.
    n = 40
    P = oracle.full_attention(g.standard_normal((n, n)), g.standard_normal((n, n)), np.eye(n))
    np.testing.assert_allclose(P.sum(1), 1.0, atol=1e-13)
    assert np.all(P > 0)
    # Row subset equals the same rows of the full computation.
    Kr = g.standard_normal((N, d))
    rows = np.array([0, 17, 199, 5])
    np.testing.assert_allclose(oracle.full_attention(Q, Kr, V, rows=rows), oracle.full_attention(Q, Kr, V)[rows], rtol=1e-13)


def _mlp_params(g, d, L, zero_out=False):
    W1, b1 = g.standard_normal((L, 2 * d)) * 0.3, g.standard_normal(L) * 0.1
    W2, b2 = g.standard_normal((d, L)) * 0.3, g.standard_normal(d) * 0.1
    if zero_out:
        W2, b2 = np.zeros_like(W2), np.zeros_like(b2)
    return W1, b1, W2, b2


def test_surrogate_without_correction_is_single_query_attention():
    g = np.random.default_rng(2)
    N, d, L = 500, 64, 64
    V = g.standard_normal((N, d))
    r = oracle.softmax(g.standard_normal(N) * 4)
    y, C = oracle.surrogate_attention(V, r, _mlp_params(g, d, L), _mlp_params(g, d, L, zero_out=True))
    # delta = 0 -> y = C_h = r_h V_h for every token.
    np.testing.assert_allclose(C, (V * r[:, None]).sum(0), rtol=1e-12)
    np.testing.assert_allclose(y, np.tile(C, (N, 1)), rtol=1e-12)
    # One-hot routing vector: C_h is that token's value.
    onehot = np.zeros(N)
    onehot[123] = 1.0
    _, C1 = oracle.surrogate_attention(V, onehot, _mlp_params(g, d, L), _mlp_params(g, d, L, zero_out=True))
    np.testing.assert_array_equal(C1, V[123])


def test_surrogate_concatenation_order_gate_and_activation():
    # z = [v_i, C_h].  MLP_delta's first layer picks the v half (W1 = [I | 0]), its
    # second layer is the identity; MLP_gamma has a zero output layer, so
    # gamma = sigma(0) = 1/2.  Then y_i = C_h + 1/2 * v_i * Phi(v_i) channel-wise.
    g = np.random.default_rng(3)
    N, d = 64, 8
    V = g.standard_normal((N, d)) * 2
    r = oracle.softmax(g.standard_normal(N))
    C = (V * r[:, None]).sum(0)
    I = np.eye(d)
    pick_v = (np.concatenate([I, np.zeros((d, d))], 1), np.zeros(d), I, np.zeros(d))
    pick_c = (np.concatenate([np.zeros((d, d)), I], 1), np.zeros(d), I, np.zeros(d))
    gamma0 = (np.zeros((d, 2 * d)), np.zeros(d), np.zeros((d, d)), np.zeros(d))
    y, _ = oracle.surrogate_attention(V, r, gamma0, pick_v)
    np.testing.assert_allclose(y, C + 0.5 * V * scipy.stats.norm.cdf(V), rtol=1e-12, atol=1e-13)
    # Picking the context half makes the correction identical for every token.
    y2, _ = oracle.surrogate_attention(V, r, gamma0, pick_c)
    np.testing.assert_allclose(y2, np.tile(C + 0.5 * C * scipy.stats.norm.cdf(C), (N, 1)), rtol=1e-12)
    # A gate MLP whose output bias is b gives gamma = expit(b) channel-wise.
    b = np.linspace(-3, 3, d)
    gamma_b = (np.zeros((d, 2 * d)), np.zeros(d), np.zeros((d, d)), b)
    y3, _ = oracle.surrogate_attention(V, r, gamma_b, pick_v)
    np.testing.assert_allclose(y3, C + scipy.special.expit(b) * V * scipy.stats.norm.cdf(V), rtol=1e-12, atol=1e-13)


def test_surrogate_rows_subset():
    g = np.random.default_rng(4)
    V = g.standard_normal((100, 64))
    r = oracle.softmax(g.standard_normal(100))
    mg, md = _mlp_params(g, 64, 64), _mlp_params(g, 64, 64)
    full, _ = oracle.surrogate_attention(V, r, mg, md)
    rows = [3, 99, 0]
    sub, _ = oracle.surrogate_attention(V, r, mg, md, rows=rows)
    np.testing.assert_allclose(sub, full[rows], rtol=1e-12, atol=1e-14)


def test_mean_pooling_closed_forms():
    g = np.random.default_rng(5)
    v = g.standard_normal(64)
    Vc = np.tile(v, (333, 1))
    y, mu = oracle.mean_pooling(Vc)
    np.testing.assert_allclose(y, Vc, rtol=1e-14)
    A, B = g.standard_normal((50, 64)), g.standard_normal((50, 64))
    ya, _ = oracle.mean_pooling(A)
    yb, _ = oracle.mean_pooling(B)
    yab, _ = oracle.mean_pooling(2 * A - 3 * B)
    np.testing.assert_allclose(yab, 2 * ya - 3 * yb, rtol=1e-12, atol=1e-13)
    np.testing.assert_allclose(ya[0], A.mean(0), rtol=1e-13)


def test_max_attention_saliency_closed_forms():
    """MaxAttn saliency s^attn = max_{i,j} A_ij (§3 and the appendix's saliency metrics)."""
    g = np.random.default_rng(11)
    N, d = 50, 64
    # identical keys: every row of A is uniform, s = 1/N
    K = np.tile(g.standard_normal(d), (N, 1))
    assert abs(oracle.max_attention_saliency(g.standard_normal((7, d)), K) - 1.0 / N) < 1e-15
    # one key scored gap g above the N-1 others for a single query: s = 1 / (1 + (N-1) e^-gap)
    q = np.zeros((1, d)); q[0, 0] = 8.0  # scores = k[:, 0] (q.k / sqrt(64) = k0)
    K = np.zeros((N, d)); K[3, 0] = 2.5
    want = 1.0 / (1.0 + (N - 1) * np.exp(-2.5))
    assert abs(oracle.max_attention_saliency(q, K) - want) < 1e-14
    # several queries: the maximum over rows is taken (the peaked row wins over uniform ones)
    Q = np.vstack([np.zeros((5, d)), q])
    assert abs(oracle.max_attention_saliency(Q, K) - want) < 1e-14


def test_max_attention_saliency_brute_force_and_invariances():
    g = np.random.default_rng(12)
    n, d = 9, 64
    Q, K = 2 * g.standard_normal((n, d)), 2 * g.standard_normal((n + 4, d))
    # brute force: each entry of A from its own numerator and denominator
    best = 0.0
    for i in range(n):
        z = [float(np.dot(Q[i], K[j]) / 8.0) for j in range(n + 4)]
        den = sum(np.exp(v) for v in z)
        best = max(best, max(np.exp(v) / den for v in z))
    s = oracle.max_attention_saliency(Q, K, chunk=4)
    assert abs(s - best) < 1e-13
    # invariant under permutations of queries and of keys; bounded by [1/N_k, 1]
    assert abs(oracle.max_attention_saliency(Q[::-1], K[g.permutation(n + 4)]) - s) < 1e-13
    assert 1.0 / (n + 4) <= s <= 1.0
    # scaling the scores up sharpens A: s is non-decreasing in the score scale
    assert oracle.max_attention_saliency(3 * Q, K) >= s


# ------------------------------------------------------------------ §5 ablation variants
def _mlps(g, d=64, L=64, delta_zero=False):
    def mlp(zero=False):
        W1 = g.standard_normal((L, 2 * d)) * 0.1
        b1 = g.standard_normal(L) * 0.1
        W2 = (0 if zero else 1) * g.standard_normal((d, L)) * 0.1
        b2 = (0 if zero else 1) * g.standard_normal(d) * 0.1
        return W1, b1, W2, b2
    return mlp(), mlp(delta_zero)


def test_surrogate_mean_context_equals_uniform_routing_vector():
    """Context replaced by the mean-pooled value vector = the surrogate with r_h = 1/N."""
    g = np.random.default_rng(31)
    N, d = 40, 64
    V = g.standard_normal((N, d))
    mg, md = _mlps(g)
    r = g.dirichlet(np.ones(N))
    got, C = oracle.surrogate_attention(V, r, mg, md, mean_context=True)
    want, Cw = oracle.surrogate_attention(V, np.full(N, 1.0 / N), mg, md)
    np.testing.assert_allclose(C, V.mean(0), rtol=1e-13, atol=1e-15)
    np.testing.assert_allclose(got, want, rtol=1e-12, atol=1e-14)


def test_surrogate_without_residual_equals_zero_delta_mlp():
    """No token-wise residual correction: y_i = C_h, the same as a zero MLP_delta."""
    g = np.random.default_rng(32)
    N, d = 33, 64
    V = g.standard_normal((N, d))
    r = g.dirichlet(np.ones(N))
    mg, md = _mlps(g, delta_zero=True)
    got, C = oracle.surrogate_attention(V, r, mg, md, residual=False, rows=np.arange(5, 20))
    want, _ = oracle.surrogate_attention(V, r, mg, md, rows=np.arange(5, 20))
    np.testing.assert_allclose(got, np.tile(r @ V, (15, 1)), rtol=1e-13, atol=1e-15)
    np.testing.assert_allclose(got, want, rtol=1e-12, atol=1e-14)


def test_elu_feature_map():
    x = np.array([-30.0, -2.0, -1e-9, 0.0, 1e-9, 0.5, 3.0])
    want = np.array([np.exp(-30.0), np.exp(-2.0), np.exp(-1e-9), 1.0, 1.0 + 1e-9, 1.5, 4.0])
    np.testing.assert_allclose(oracle.elu_feature_map(x), want, rtol=1e-15)
    assert np.all(oracle.elu_feature_map(x) > 0)


def test_linear_attention_closed_forms_and_brute_force():
    g = np.random.default_rng(33)
    N, d = 23, 64
    Q, K, V = g.standard_normal((N, d)), g.standard_normal((N, d)), g.standard_normal((N, d))
    # constant V rows give V back; identical keys give the mean of V for every query
    c = g.standard_normal(d)
    np.testing.assert_allclose(oracle.linear_attention(Q, K, np.tile(c, (N, 1))), np.tile(c, (N, 1)), rtol=1e-12)
    np.testing.assert_allclose(oracle.linear_attention(Q, np.tile(K[0], (N, 1)), V), np.tile(V.mean(0), (N, 1)),
                               rtol=1e-11, atol=1e-13)
    # brute force, one pair at a time, from the elementwise feature map
    phi = lambda x: x + 1.0 if x > 0 else np.exp(x)
    out = oracle.linear_attention(Q, K, V, chunk=5)
    for i in (0, 7, N - 1):
        w = np.array([sum(phi(Q[i, t]) * phi(K[j, t]) for t in range(d)) for j in range(N)])
        np.testing.assert_allclose(out[i], (w @ V) / w.sum(), rtol=1e-11)
    # the factored order the kernels use, phi(Q) (phi(K)^T V) / (phi(Q) phi(K)^T 1), is the same map
    fQ, fK = oracle.elu_feature_map(Q), oracle.elu_feature_map(K)
    np.testing.assert_allclose(out, (fQ @ (fK.T @ V)) / (fQ @ fK.sum(0))[:, None], rtol=1e-11)
    # positive weights: every output lies within the range of V's column
    assert np.all(out <= V.max(0) + 1e-12) and np.all(out >= V.min(0) - 1e-12)
    # rows subset
    np.testing.assert_allclose(oracle.linear_attention(Q, K, V, rows=[3, 9]), out[[3, 9]], rtol=1e-13)
