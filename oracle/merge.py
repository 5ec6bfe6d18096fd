"""Token merging (ToMe) around a block's attention, float64.  Test infrastructure only.

The paper combines VGGT-Prime with the token merging of FastVGGT (75 % and 90 % of the tokens
merged) and defines nothing further; this is the library's reading (vp_merge_options):
destinations are the special tokens of every view, every token of the first view and every
stride-th patch token of the other views; each source joins the destination whose head-mean
key, as a unit vector, is most similar to its own (ToMe's bipartite matching with the keys
as the metric); a merged token is the mean of its members; the attention output of a merged
token goes back to all of them (unmerge).  Parity unpinned to the paper (it prints nothing
on the merging); the tests pin these functions to hand-built cases and conservation laws.
"""
from __future__ import annotations

import numpy as np


def destinations(N: int, tokens_per_view: int, patch_start: int, stride: int):
    """(row_of [N]: merged row of each destination, -1 for sources; dst_tok [Np]: the token
    of each merged row).  Merged rows follow token order."""
    t = np.arange(N) % tokens_per_view
    v = np.arange(N) // tokens_per_view
    is_dst = (v == 0) | (t < patch_start) | ((t - patch_start) % stride == 0)
    dst_tok = np.nonzero(is_dst)[0]
    row_of = np.full(N, -1, np.int64)
    row_of[dst_tok] = np.arange(len(dst_tok))
    return row_of, dst_tok


def key_metric(Xt, lw):
    """Unit head-mean keys of the LN1 output, in exact arithmetic: k_i = mean_h (Xt_i W_K,h^T
    + b_K,h), m_i = k_i / |k_i| (0 for a zero key).  The metric is no storage point of the
    block (the paper fixes no precision for it), so nothing here is rounded to bf16."""
    H = lw["r_W"].shape[0]
    D = Xt.shape[1]
    wk = lw["w_qkv"][D:2 * D].reshape(H, 64, D)
    bk = lw["b_qkv"][D:2 * D].reshape(H, 64)
    k = np.asarray(Xt, np.float64) @ wk.mean(axis=0).T + bk.mean(axis=0)
    norm = np.sqrt(np.sum(k * k, axis=1, keepdims=True))
    return np.where(norm > 0, k / np.where(norm > 0, norm, 1.0), 0.0)


def match(m, row_of, dst_tok):
    """assign [N]: each destination's own row; for a source, the row of the destination of
    largest m_i . m_j (ties: the lowest row).  Also returns the scores [N, Np]."""
    scores = m @ m[dst_tok].T
    assign = np.argmax(scores, axis=1)  # first maximum = lowest row
    assign = np.where(row_of >= 0, row_of, assign)
    return assign, scores


def merge_tokens(Xt, assign, n_rows):
    """Mean of each merged row's members: [Np, D]."""
    Xt = np.asarray(Xt, np.float64)
    sums = np.zeros((n_rows, Xt.shape[1]))
    np.add.at(sums, assign, Xt)
    counts = np.bincount(assign, minlength=n_rows)
    return sums / counts[:, None]
