"""Positional information and qk-norm of the QKV step, float64.  Test infrastructure only.

Algorithm 1 step (2) computes Q, K, V from X~ "with positional information P"; the paper
does not define P.  The reading here (the library's vp_qk_options) is the positional scheme
of the VGGT backbone that VGGT-Prime modifies: a per-head LayerNorm of q and k over their d
channels (qk-norm), then a two-dimensional rotary position embedding (RoFormer's rotation
applied once per image axis) at the token's patch position inside its view.  Special tokens
(camera, registers) sit at position (0, 0), which leaves them unrotated.  Parity unpinned
to the paper (it prints nothing on P); the tests pin these functions to the mathematics:
norms preserved, axis separation, scores that depend on relative positions only, and
LayerNorm against the library routine.
"""
from __future__ import annotations

import numpy as np

from .numerics import layer_norm


def token_positions(N: int, tokens_per_view: int, patch_start: int, grid_w: int):
    """(row, column) position of each of N tokens, views concatenated: (0, 0) for the
    patch_start special tokens of a view, (r + 1, c + 1) for its patch r * grid_w + c."""
    t = np.arange(N) % tokens_per_view - patch_start
    py = np.where(t >= 0, t // grid_w + 1, 0)
    px = np.where(t >= 0, t % grid_w + 1, 0)
    return py.astype(np.int64), px.astype(np.int64)


def rope_2d(x, py, px, base: float):
    """Two-dimensional rotary embedding of x [N, d] (d divisible by 4): channels [0, d/2)
    turn with the row position py, [d/2, d) with the column position px.  Within a half of
    h = d/2 channels, channel i and channel i + h/2 (i < h/2) form a plane turned by the
    angle pos * base^(-2 i / h): (a, b) -> (a cos - b sin, b cos + a sin)."""
    x = np.array(x, dtype=np.float64)
    d = x.shape[1]
    h = d // 2
    q = h // 2
    theta = base ** (-2.0 * np.arange(q) / h)
    out = x.copy()
    for half, pos in ((0, py), (1, px)):
        ang = np.asarray(pos, np.float64)[:, None] * theta[None, :]
        c, s = np.cos(ang), np.sin(ang)
        a = x[:, half * h: half * h + q]
        b = x[:, half * h + q: half * h + h]
        out[:, half * h: half * h + q] = a * c - b * s
        out[:, half * h + q: half * h + h] = b * c + a * s
    return out


def qk_transform(x, norm, eps, positions, base):
    """One head's q (or k) [N, d]: LayerNorm over d with (gamma, beta) = norm (None: skip),
    then rope_2d at positions = (py, px) (None: skip)."""
    x = np.asarray(x, np.float64)
    if norm is not None:
        x = layer_norm(x, norm[0], norm[1], eps)
    if positions is not None:
        x = rope_2d(x, positions[0], positions[1], base)
    return x
