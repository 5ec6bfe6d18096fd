"""CPU oracle for VGGT-Prime's mixture-of-heads global attention.

TEST INFRASTRUCTURE ONLY.  This package is a plain, slow, float64 restatement
of the method as the paper defines it (§4.1 head saliency, §4.2 head routing,
§4.3 surrogate attention, Algorithm 1 in App. B).  It exists to check the CUDA
path; only ``tests/``, ``__graft_entry__.smoke()`` and the CPU-baseline leg of
``bench.py`` may import it.  The library never calls it, and it shares no code
with the CUDA path: the only common module is ``synth`` (seeded random inputs).

Precision: every step runs in float64.  Where the library stores a tensor in
bf16 (QKV, the head outputs Y, the layer output, and inside the block the LN2
output, the residual stream and the FFN hidden layer) the oracle
rounds its float64 values to the nearest bf16 at the same point, through the
``materialize`` argument; pins pass ``materialize=None`` to compare against
textbook formulations without those storage roundings.  Mode decisions compare
the saliency rounded to float32 with float32 thresholds, as the library does.

Parity status: the router (§4.1), routing rule (§4.2), full and mean modes
(Algorithm 1), the MaxAttn saliency (§3, appendix) and the block are pinned by tests in tests/test_oracle_*.py.  Two
choices the paper leaves open are pinned only to the stated reading, not to a
printed value: the scale of the routing attention (taken as beta_h / sqrt(d),
beta_h = 1, like full attention) and the shape of MLP_gamma / MLP_delta
(Linear(2d -> 64) -> GELU -> Linear(64 -> d), hidden width 64 from App. B).
"""
from .numerics import round_bf16, bf16_bits_to_f64, sigmoid, gelu, softmax, layer_norm
from .router import (pooling_logits, attention_pool, routing_vector, saliency,
                     select_mode, route_heads, bin_heads, MODE_MEAN, MODE_SURROGATE,
                     MODE_FULL, Q_TILE)
from .modes import (full_attention, surrogate_attention, mean_pooling, surrogate_mlp,
                    max_attention_saliency, elu_feature_map, linear_attention)
from .layer import (qkv_projection, head_router, moh_attention, global_block,
                    global_stack, load_layer, VARIANTS)
from .position import token_positions, rope_2d, qk_transform
from .merge import destinations, key_metric, match, merge_tokens

__all__ = [
    "round_bf16", "bf16_bits_to_f64", "sigmoid", "gelu", "softmax", "layer_norm",
    "pooling_logits", "attention_pool", "routing_vector", "saliency", "select_mode",
    "route_heads", "bin_heads", "MODE_MEAN", "MODE_SURROGATE", "MODE_FULL", "Q_TILE",
    "full_attention", "surrogate_attention", "mean_pooling", "surrogate_mlp",
    "max_attention_saliency", "elu_feature_map", "linear_attention", "VARIANTS",
    "qkv_projection", "head_router", "moh_attention", "global_block", "global_stack",
    "token_positions", "rope_2d", "qk_transform", "destinations", "key_metric", "match",
    "merge_tokens",
    "load_layer",
]
