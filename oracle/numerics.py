"""Scalar building blocks of the oracle (float64).  Test infrastructure only.

Each function is the textbook definition; nothing is fused or reordered.
"""
from __future__ import annotations

import numpy as np
from scipy.special import erf

# Largest finite bf16 value: (2 - 2^-7) * 2^127.
BF16_MAX = (2.0 - 2.0 ** -7) * 2.0 ** 127


def round_bf16(x) -> np.ndarray:
    """Round float64 values to the nearest bf16 value, ties to even.

    bf16 keeps 8 significant bits (1 implicit + 7 stored) and float32's
    exponent range; below 2^-126 the spacing stays 2^-133 (subnormals).
    The result is returned as float64 (exactly representable).

    In bf16's normal range the rounding is done on the float64 bit pattern: of the 52
    stored mantissa bits, bf16 keeps the top 7, so the low 45 bits are dropped after
    adding half of their weight (2^44), minus one unless the lowest kept bit is odd (ties
    go to the even neighbour); a carry out of the mantissa moves to the next binade, as it
    should.  Below 2^-126 the value is rounded at the fixed spacing 2^-133 instead.
    """
    x = np.ascontiguousarray(np.asarray(x, dtype=np.float64))
    b = x.view(np.uint64)
    keep = (b >> np.uint64(45)) & np.uint64(1)
    y = ((b + (np.uint64((1 << 44) - 1) + keep)) >> np.uint64(45) << np.uint64(45)).view(np.float64)
    small = np.abs(x) < 2.0 ** -126
    if np.any(small):  # bf16 subnormals: multiples of 2^-133 (rint: half to even)
        y = np.where(small, np.ldexp(np.rint(np.ldexp(x, 133)), -133), y)
    y = np.where(np.isfinite(x), y, x)
    over = np.abs(y) > BF16_MAX
    if np.any(over):
        y = np.where(over, np.copysign(np.inf, x), y)
    return y


def bf16_bits_to_f64(u) -> np.ndarray:
    """Decode bf16 bit patterns (uint16) to float64."""
    u = np.asarray(u, dtype=np.uint16)
    with np.errstate(invalid="ignore"):
        return (u.astype(np.uint32) << 16).view(np.float32).astype(np.float64)


def sigmoid(x):
    """sigma(x) = 1 / (1 + exp(-x))."""
    x = np.asarray(x, dtype=np.float64)
    with np.errstate(over="ignore"):
        return 1.0 / (1.0 + np.exp(-x))


def gelu(x):
    """GELU, exact (erf) form: x * Phi(x) = 0.5 x (1 + erf(x / sqrt 2))."""
    x = np.asarray(x, dtype=np.float64)
    return 0.5 * x * (1.0 + erf(x / np.sqrt(2.0)))


def softmax(v, axis=-1):
    """exp(v_i) / sum_j exp(v_j), evaluated with the maximum subtracted."""
    v = np.asarray(v, dtype=np.float64)
    m = np.max(v, axis=axis, keepdims=True)
    p = np.exp(v - m)
    return p / np.sum(p, axis=axis, keepdims=True)


def layer_norm(x, gamma, beta, eps: float = 1e-6):
    """LN over the last axis: (x - mean) / sqrt(var + eps) * gamma + beta,
    with the biased (1/D) variance."""
    x = np.asarray(x, dtype=np.float64)
    mu = x.mean(axis=-1, keepdims=True)
    var = ((x - mu) ** 2).mean(axis=-1, keepdims=True)
    return (x - mu) / np.sqrt(var + eps) * np.asarray(gamma, np.float64) + np.asarray(beta, np.float64)
