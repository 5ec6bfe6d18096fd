"""Shared helpers for the parity tests: seeded inputs (from ``synth``), calls through the
C ABI (``paper_2609_23733_gb300.binding``), and the oracle's expected values."""
from __future__ import annotations

import numpy as np

import oracle
import synth

# Parity bar for bf16 outputs with fp32 accumulation.
MAX_ABS = 2e-2
MEAN_ABS = 2e-3
# Guard band: oracle saliencies this close (relative) to a threshold are not used for
# exact route comparisons (the two sides reduce in different orders).
GUARD = 1e-3


# Both sides round a stored bf16 value independently; a value within rounding noise of a
# rounding boundary may land one bf16 step (2^-7 relative at most) apart.  ``rel`` adds that
# step for large-magnitude outputs (the residual stream), where one step exceeds MAX_ABS.
BF16_STEP = 2.0 ** -7


def compare(got, want, max_abs=MAX_ABS, mean_abs=MEAN_ABS, rel=0.0, what=""):
    got = np.asarray(got, np.float64)
    want = np.asarray(want, np.float64)
    assert got.shape == want.shape, (what, got.shape, want.shape)
    assert np.all(np.isfinite(got)), f"{what}: non-finite values"
    err = np.abs(got - want)
    excess = err - (max_abs + rel * np.abs(want))
    mx, mn = float(err.max(initial=0.0)), float(err.mean()) if err.size else 0.0
    assert float(excess.max(initial=-1.0)) <= 0 and mn <= mean_abs, \
        f"{what}: max-abs {mx:.3e} mean-abs {mn:.3e} (worst excess {float(excess.max(initial=0)):.3e})"
    return mx, mn


def outside_guard(s, tau_low=0.01, tau_high=0.20, guard=GUARD):
    s = np.asarray(s, np.float64)
    return (np.abs(s - tau_low) > guard * tau_low) & (np.abs(s - tau_high) > guard * tau_high)


def calibrate_beta(qkv, lw, h, target, lo=1e-3, hi=1e7, iters=80):
    """Routing temperature beta_h that puts the oracle's saliency of head h at ``target``
    (bisection in log space; s_h is non-decreasing in beta_h)."""
    Q_h, K_h = qkv[:, 0, h], qkv[:, 1, h]
    _, q_pool = oracle.attention_pool(Q_h, lw["r_W"][h], lw["r_U"][h], lw["r_w"][h], lw["r_bW"][h], lw["r_bU"][h])
    d = Q_h.shape[1]
    for _ in range(iters):
        mid = np.sqrt(lo * hi)
        s = oracle.saliency(oracle.routing_vector(q_pool, K_h, mid / np.sqrt(d)))
        if s < target:
            lo = mid
        else:
            hi = mid
    return float(np.sqrt(lo * hi))


# Saliency targets used to steer heads into each band (geometric middles of the bands).
TARGET_FULL = 0.5
TARGET_SURROGATE = float(np.sqrt(0.01 * 0.2))


def calibrated_layer(seed, N, mix, H=16, D=1024, bias_std=0.0, block=False):
    """Tokens and one layer's weights whose routers are steered (per-head beta) so that
    head h lands in mode mix[h] (None = leave beta at 1).  Returns (x_bits, w, lw64)."""
    g = synth.rng(seed)
    w = synth.make_layer_weights(g, D=D, H=H, d=D // H, block=block, bias_std=bias_std)
    x_bits = synth.make_tokens(seed, N, D)
    lw = oracle.load_layer(w)
    X = oracle.bf16_bits_to_f64(x_bits)
    if block:
        X = oracle.round_bf16(oracle.layer_norm(X, lw["ln1_g"], lw["ln1_b"], 1e-6))
    qkv = oracle.qkv_projection(X, lw)
    beta = np.ones(H, np.float32)
    for h, m in enumerate(mix):
        if m == synth.MODE_FULL:
            beta[h] = calibrate_beta(qkv, lw, h, TARGET_FULL)
        elif m == synth.MODE_SURROGATE:
            beta[h] = calibrate_beta(qkv, lw, h, TARGET_SURROGATE)
    w["r_beta"] = beta
    lw["r_beta"] = beta.astype(np.float64)
    return x_bits, w, lw
