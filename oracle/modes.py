"""The three computation modes of a routed head, float64.  Test infrastructure only.

Full: softmax(Q_h K_h^T / sqrt d) V_h (Algorithm 1, step 2, case s >= tau_high).
Surrogate: C_h = r_h V_h, z = [v_i, C_h], y = C_h + sigma(MLP_gamma z) (.) MLP_delta z (§4.3).
Mean: Broadcast((1/N) sum_i V_{h,i}) (Algorithm 1, step 2, case s <= tau_low).
"""
from __future__ import annotations

import numpy as np

from .numerics import gelu, sigmoid, softmax


def full_attention(Q_h, K_h, V_h, rows=None, chunk=64):
    """softmax(Q_h K_h^T / sqrt(d)) V_h for the query rows ``rows`` (all rows
    when None).  Rows are independent, so a subset is computed exactly."""
    Q_h = np.asarray(Q_h, np.float64)
    K_h = np.asarray(K_h, np.float64)
    V_h = np.asarray(V_h, np.float64)
    d = Q_h.shape[1]
    idx = np.arange(Q_h.shape[0]) if rows is None else np.asarray(rows)
    out = np.empty((len(idx), V_h.shape[1]), np.float64)
    for a in range(0, len(idx), chunk):
        sel = idx[a:a + chunk]
        P = softmax((Q_h[sel] @ K_h.T) / np.sqrt(d), axis=1)
        out[a:a + chunk] = P @ V_h
    return out


def max_attention_saliency(Q_h, K_h, chunk=64):
    """MaxAttn saliency of a head (§3 "Head Saliency"; defined in the appendix section on
    head saliency metrics): s_h^attn = max over all (i, j) of A_h[i, j], the largest entry
    of the post-softmax attention matrix A_h = softmax(Q_h K_h^T / sqrt(d)).  Written out as
    the definition: A_h row block by row block, then its maximum."""
    Q_h = np.asarray(Q_h, np.float64)
    K_h = np.asarray(K_h, np.float64)
    d = Q_h.shape[1]
    best = 0.0
    for a in range(0, Q_h.shape[0], chunk):
        A = softmax((Q_h[a:a + chunk] @ K_h.T) / np.sqrt(d), axis=1)
        best = max(best, float(A.max()))
    return best


def surrogate_mlp(z, W1, b1, W2, b2):
    """MLP_gamma / MLP_delta of §4.3: Linear(2d -> L) -> GELU -> Linear(L -> d).
    The paper gives the hidden width (64, App. B) but not depth or activation;
    this is the reading used throughout (one hidden layer, exact GELU)."""
    h = gelu(np.asarray(z, np.float64) @ np.asarray(W1, np.float64).T + np.asarray(b1, np.float64))
    return h @ np.asarray(W2, np.float64).T + np.asarray(b2, np.float64)


def surrogate_attention(V_h, r_h, mlp_gamma, mlp_delta, rows=None, mean_context=False,
                        residual=True):
    """§4.3.  C_h = r_h V_h; for each token z_{h,i} = [v_{h,i}, C_h];
    gamma = sigma(MLP_gamma(z)), delta = MLP_delta(z); y_i = C_h + gamma (.) delta.

    mlp_gamma / mlp_delta are (W1 [L, 2d], b1 [L], W2 [d, L], b2 [d]).
    Returns (y [rows, d], C_h [d]).

    The component ablation of §5: mean_context replaces the context vector by the mean-pooled
    value vector (C_h = (1/N) sum_i v_{h,i}); residual=False removes the token-wise residual
    correction (y_i = C_h for every token)."""
    V_h = np.asarray(V_h, np.float64)
    C = V_h.sum(axis=0) / V_h.shape[0] if mean_context else np.asarray(r_h, np.float64) @ V_h
    Vr = V_h if rows is None else V_h[np.asarray(rows)]
    if not residual:
        return np.tile(C, (Vr.shape[0], 1)), C
    z = np.concatenate([Vr, np.broadcast_to(C, Vr.shape)], axis=1)
    gamma = sigmoid(surrogate_mlp(z, *mlp_gamma))
    delta = surrogate_mlp(z, *mlp_delta)
    return C + gamma * delta, C


def elu_feature_map(x):
    """phi(x) = elu(x) + 1, the feature map of linear attention (Katharopoulos et al.,
    "Transformers are RNNs", ICML 2020, the method §5's compute-mode ablation cites)."""
    x = np.asarray(x, np.float64)
    return np.where(x > 0, x + 1.0, np.exp(np.minimum(x, 0.0)))


def linear_attention(Q_h, K_h, V_h, rows=None, chunk=64):
    """The compute-mode ablation of §5: surrogate heads replaced by (non-causal) linear
    attention.  With sim(q, k) = phi(q) . phi(k):
        y_i = sum_j sim(q_i, k_j) v_j / sum_j sim(q_i, k_j).
    Written as that definition, the similarity matrix row block by row block."""
    Q_h = np.asarray(Q_h, np.float64)
    fK = elu_feature_map(K_h)
    V_h = np.asarray(V_h, np.float64)
    idx = np.arange(Q_h.shape[0]) if rows is None else np.asarray(rows)
    out = np.empty((len(idx), V_h.shape[1]), np.float64)
    for a in range(0, len(idx), chunk):
        sel = idx[a:a + chunk]
        A = elu_feature_map(Q_h[sel]) @ fK.T
        out[a:a + chunk] = (A @ V_h) / A.sum(axis=1, keepdims=True)
    return out


def mean_pooling(V_h, n_rows=None):
    """Broadcast((1/N) sum_i V_{h,i}) to ``n_rows`` rows (N when None)."""
    V_h = np.asarray(V_h, np.float64)
    mu = V_h.sum(axis=0) / V_h.shape[0]
    return np.broadcast_to(mu, (V_h.shape[0] if n_rows is None else n_rows, V_h.shape[1])).copy(), mu
