"""Router of VGGT-Prime, float64.  Test infrastructure only.

§4.1 (head saliency): gated attention pooling of the queries, single-query
attention of the pooled query over all keys, saliency = max routing weight.
§4.2 (head routing): two thresholds split heads into full / surrogate / mean.
"""
from __future__ import annotations

import numpy as np

from .numerics import sigmoid, softmax

MODE_MEAN, MODE_SURROGATE, MODE_FULL = 0, 1, 2
Q_TILE = 128          # query rows per work item of a full-mode head


def pooling_logits(Q_h, W_h, U_h, w_h, bW=None, bU=None):
    """§4.1, argument of the softmax that gives alpha_{h,i}:
    w_h^T ( tanh(W_h q_{h,i}) (.) sigma(U_h q_{h,i}) ) for every token i.

    Q_h [N, d]; W_h, U_h [L, d]; w_h [L]; optional biases bW, bU [L]
    (the paper writes none; zero when omitted).
    """
    Q_h = np.asarray(Q_h, np.float64)
    a = Q_h @ np.asarray(W_h, np.float64).T
    b = Q_h @ np.asarray(U_h, np.float64).T
    if bW is not None:
        a = a + np.asarray(bW, np.float64)
    if bU is not None:
        b = b + np.asarray(bU, np.float64)
    return (np.tanh(a) * sigmoid(b)) @ np.asarray(w_h, np.float64)


def attention_pool(Q_h, W_h, U_h, w_h, bW=None, bU=None, mean_pool=False):
    """§4.1: alpha_h = softmax over all N tokens of the pooling logits;
    q_pool = sum_i alpha_{h,i} q_{h,i}.  Returns (alpha [N], q_pool [d]).

    mean_pool: the component ablation of §5 ("Q-Pooling" replaced by mean pooling):
    alpha = 1/N for every token, q_pool = the mean query."""
    if mean_pool:
        N = np.asarray(Q_h).shape[0]
        alpha = np.full(N, 1.0 / N)
    else:
        alpha = softmax(pooling_logits(Q_h, W_h, U_h, w_h, bW, bU))
    return alpha, alpha @ np.asarray(Q_h, np.float64)


def routing_vector(q_pool, K_h, scale):
    """§4.1: single-query attention of q_pool over all N keys,
    r_h = softmax_j( scale * q_pool . k_j ).  The paper states no scale; the
    reading used here is scale = beta_h / sqrt(d) with beta_h = 1 by default,
    the same temperature as full attention (Algorithm 1, step 2)."""
    return softmax(scale * (np.asarray(K_h, np.float64) @ np.asarray(q_pool, np.float64)))


def saliency(r_h):
    """§4.1: s_h = max_i r_h(i)."""
    return float(np.max(r_h))


def select_mode(s, tau_low=np.float32(0.01), tau_high=np.float32(0.2)):
    """§4.2, routing equation: full if s >= tau_high, surrogate if
    tau_low < s < tau_high, mean if s <= tau_low.

    The decision is taken in float32 (the saliency rounded to float32 against
    float32 thresholds), the precision the library stores s in.  Cases are
    tested in the equation's order, full first, so s == tau_high is full and
    s == tau_low is mean; when tau_low >= tau_high (a two-way router) full
    still wins.  A NaN saliency matches no case of the equation; it is routed
    to full, the exact operator.
    """
    s32 = np.float32(s)
    if np.isnan(s32) or s32 >= np.float32(tau_high):
        return MODE_FULL
    if s32 <= np.float32(tau_low):
        return MODE_MEAN
    return MODE_SURROGATE


def route_heads(saliencies, tau_low=np.float32(0.01), tau_high=np.float32(0.2)):
    return np.array([select_mode(s, tau_low, tau_high) for s in saliencies], np.int32)


def bin_heads(modes, N, q_tile=Q_TILE):
    """Group heads by routed mode, mode 0 (mean), 1 (surrogate), 2 (full), heads
    in ascending index inside each group; offsets[m]..offsets[m+1] delimit mode
    m.  The work list enumerates (head, query tile) for every full-mode head,
    head-major, tiles ascending.  Implied by §4.2 (each head is computed by the
    operator of its case)."""
    modes = np.asarray(modes, np.int32)
    head_ids, offsets = [], [0]
    for m in (MODE_MEAN, MODE_SURROGATE, MODE_FULL):
        head_ids += [h for h in range(len(modes)) if modes[h] == m]
        offsets.append(len(head_ids))
    n_tiles = (N + q_tile - 1) // q_tile
    work = [(h, t) for h in range(len(modes)) if modes[h] == MODE_FULL for t in range(n_tiles)]
    return (np.array(head_ids, np.int32), np.array(offsets, np.int32),
            np.array(work, np.int32).reshape(-1, 2))
