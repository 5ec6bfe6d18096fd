"""Seeded synthetic inputs for the mixture-of-heads global-attention path.

This module only draws random numbers and packs them into the storage formats
the library and the oracle both read (bf16 bit patterns as ``uint16``, fp32 for
biases and norm parameters).  It holds none of the method's arithmetic, so the
CUDA path and the CPU oracle can share it without sharing any computation.

Shapes follow VGGT's aggregator: model width D = 1024, H = 16 heads of d = 64,
router and surrogate hidden width L = 64 (App. B, "Hyperparameters"), tokens per
view P = 1 camera + 4 register + patch tokens, views concatenated along the
token axis (§3; Algorithm 1 takes all S*P tokens of all views at once).
The paper's datasets are not available; these draws stand in for them.
"""
from __future__ import annotations

from dataclasses import dataclass, field

import numpy as np

D_MODEL = 1024
N_HEADS = 16
HEAD_DIM = 64
HIDDEN = 64          # router / surrogate hidden width (App. B)
FFN_RATIO = 4
TAU_LOW = 0.01       # §4.2 and App. B
TAU_HIGH = 0.20

MODE_MEAN, MODE_SURROGATE, MODE_FULL = 0, 1, 2


def tokens_per_view(image_px: int, patch: int = 14) -> int:
    """1 camera + 4 register tokens + (image_px / patch)^2 patch tokens."""
    g = image_px // patch
    return g * g + 5


@dataclass(frozen=True)
class Workload:
    name: str
    views: int
    image_px: int
    layers: int
    seed: int
    routing: str                  # "natural", "calibrated", "forced_sweep", "paper_mix"
    full_fractions: tuple = field(default=())

    @property
    def P(self) -> int:
        return tokens_per_view(self.image_px)

    @property
    def N(self) -> int:
        return self.views * self.P


# The five workloads: single layers at S=4 (224 px) and S=8 (518 px), 24-layer
# stacks at S=32 and S=100 (518 px), and a routing-mix sweep at S=64.
WORKLOADS = {
    "s4_layer": Workload("s4_layer", 4, 224, 1, 0, "natural"),
    "s8_layer_biased": Workload("s8_layer_biased", 8, 518, 1, 1, "calibrated"),
    "s32_stack": Workload("s32_stack", 32, 518, 24, 2, "natural"),
    "s100_stack": Workload("s100_stack", 100, 518, 24, 3, "paper_mix"),
    "s64_mix_sweep": Workload("s64_mix_sweep", 64, 518, 1, 4, "forced_sweep",
                              (0.0, 0.25, 0.5, 1.0)),
}


def rng(seed: int) -> np.random.Generator:
    return np.random.Generator(np.random.PCG64(seed))


def f32_to_bf16_bits(x) -> np.ndarray:
    """Pack float values into bf16 bit patterns (round to nearest even)."""
    b = np.ascontiguousarray(np.asarray(x, dtype=np.float32)).view(np.uint32)
    # Finite values stay below 0xFF800000, so the rounding add cannot wrap in 32 bits.
    b = (b + (np.uint32(0x7FFF) + ((b >> np.uint32(16)) & np.uint32(1)))) >> np.uint32(16)
    return b.astype(np.uint16)


def bf16_bits_to_f32(u) -> np.ndarray:
    """Unpack bf16 bit patterns into float32 values (exact)."""
    u = np.asarray(u, dtype=np.uint16)
    return (u.astype(np.uint32) << 16).view(np.float32)


def xavier_uniform(g: np.random.Generator, fan_out: int, fan_in: int, batch=()) -> np.ndarray:
    """Xavier/Glorot uniform draw for a weight of shape batch + (fan_out, fan_in)."""
    bound = np.sqrt(6.0 / (fan_in + fan_out))
    return g.uniform(-bound, bound, size=tuple(batch) + (fan_out, fan_in)).astype(np.float32)


def make_tokens(seed: int, N: int, D: int = D_MODEL) -> np.ndarray:
    """Activations X ~ N(0, 1), [N, D], as bf16 bits."""
    g = rng(seed)
    return f32_to_bf16_bits(g.standard_normal((N, D), dtype=np.float32))


def make_qk_norm_weights(g: np.random.Generator, *, d: int = HEAD_DIM, jitter: float = 0.1,
                         bias_std: float = 0.05) -> dict:
    """qk-norm parameters (per-channel LayerNorm scale and shift of q and k, shared by the
    heads), float32: q_norm_g, q_norm_b, k_norm_g, k_norm_b."""
    w = {}
    for t in ("q", "k"):
        w[f"{t}_norm_g"] = (1.0 + jitter * g.standard_normal(d)).astype(np.float32)
        w[f"{t}_norm_b"] = (bias_std * g.standard_normal(d)).astype(np.float32)
    return w


def make_layer_weights(g: np.random.Generator, *, D: int = D_MODEL, H: int = N_HEADS,
                       d: int = HEAD_DIM, L: int = HIDDEN, block: bool = False,
                       bias_std: float = 0.0, norm_jitter: float = 0.0) -> dict:
    """One layer's parameters in a fixed draw order.

    Matrices are bf16 bits in the nn.Linear layout (out_features, in_features);
    biases, LayerNorm and LayerScale parameters are float32.  ``bias_std`` and
    ``norm_jitter`` default to the zero-bias / unit-scale initialisation; tests
    turn them on so that every bias and scale path carries signal.
    """
    assert H * d == D

    def bias(*shape):
        if bias_std == 0.0:
            return np.zeros(shape, np.float32)
        return (bias_std * g.standard_normal(shape)).astype(np.float32)

    w = {}
    # Projections of the attention block: QKV rows ordered (3, H, d), output (D, D).
    w["w_qkv"] = f32_to_bf16_bits(xavier_uniform(g, 3 * D, D))
    w["b_qkv"] = bias(3 * D)
    w["w_o"] = f32_to_bf16_bits(xavier_uniform(g, D, D))
    w["b_o"] = bias(D)
    # Router, per head: W_h, U_h in R^{L x d}, w_h in R^L (§4.1).
    w["r_W"] = f32_to_bf16_bits(xavier_uniform(g, L, d, (H,)))
    w["r_U"] = f32_to_bf16_bits(xavier_uniform(g, L, d, (H,)))
    w["r_w"] = f32_to_bf16_bits(xavier_uniform(g, 1, L, (H,)).reshape(H, L))
    w["r_bW"] = bias(H, L)
    w["r_bU"] = bias(H, L)
    w["r_beta"] = np.ones(H, np.float32)
    # Surrogate MLPs, per head: Linear(2d -> L) -> GELU -> Linear(L -> d) (§4.3).
    for m in ("g", "d"):
        w[f"s_{m}1_w"] = f32_to_bf16_bits(xavier_uniform(g, L, 2 * d, (H,)))
        w[f"s_{m}1_b"] = bias(H, L)
        w[f"s_{m}2_w"] = f32_to_bf16_bits(xavier_uniform(g, d, L, (H,)))
        w[f"s_{m}2_b"] = bias(H, d)
    if block:
        def norm_scale(n):
            if norm_jitter == 0.0:
                return np.ones(n, np.float32)
            return (1.0 + norm_jitter * g.standard_normal(n)).astype(np.float32)
        w["ln1_g"] = norm_scale(D)
        w["ln1_b"] = bias(D)
        w["ls1"] = norm_scale(D)
        w["ln2_g"] = norm_scale(D)
        w["ln2_b"] = bias(D)
        w["w_fc1"] = f32_to_bf16_bits(xavier_uniform(g, FFN_RATIO * D, D))
        w["b_fc1"] = bias(FFN_RATIO * D)
        w["w_fc2"] = f32_to_bf16_bits(xavier_uniform(g, D, FFN_RATIO * D))
        w["b_fc2"] = bias(D)
        w["ls2"] = norm_scale(D)
    return w


def make_stack_weights(seed: int, n_layers: int, **kw) -> list:
    g = rng(seed + 1000)
    return [make_layer_weights(g, block=True, **kw) for _ in range(n_layers)]


def forced_mix(n_heads: int, full_fraction: float) -> np.ndarray:
    """Forced routes for the mix sweep: heads 0..n_full-1 full, the rest
    alternate surrogate / mean by parity of (h - n_full)."""
    n_full = int(round(full_fraction * n_heads))
    m = np.empty(n_heads, np.int32)
    for h in range(n_heads):
        if h < n_full:
            m[h] = MODE_FULL
        else:
            m[h] = MODE_SURROGATE if (h - n_full) % 2 == 0 else MODE_MEAN
    return m


# Average routing distribution of the trained router over seven datasets
# (App. E.2, routing-distribution table): mean 50.0 %, surrogate 42.2 %,
# full 7.8 % of all heads.
PAPER_MIX = {"mean": 0.500, "surrogate": 0.422, "full": 0.078}


def paper_mix_modes(n_layers: int, n_heads: int = N_HEADS) -> np.ndarray:
    """[n_layers, n_heads] routes whose totals match PAPER_MIX as closely as
    integers allow, spread evenly over layers (a deterministic schedule)."""
    total = n_layers * n_heads
    n_full = int(round(PAPER_MIX["full"] * total))
    n_mean = int(round(PAPER_MIX["mean"] * total))
    modes = np.full((n_layers, n_heads), MODE_SURROGATE, np.int32)
    # Distribute full heads round-robin over layers, placed at rotating head
    # indices so that every head slot sees each mode somewhere in the stack.
    full_per_layer = [n_full // n_layers + (1 if l < n_full % n_layers else 0) for l in range(n_layers)]
    mean_per_layer = [n_mean // n_layers + (1 if l < n_mean % n_layers else 0) for l in range(n_layers)]
    for l in range(n_layers):
        order = [(l * 5 + k) % n_heads for k in range(n_heads)]
        for k in range(full_per_layer[l]):
            modes[l, order[k]] = MODE_FULL
        for k in range(mean_per_layer[l]):
            modes[l, order[full_per_layer[l] + k]] = MODE_MEAN
    return modes
