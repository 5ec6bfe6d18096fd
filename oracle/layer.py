"""Routed global-attention layer and Algorithm 1's block, float64.  Test infrastructure only.

moh_attention: Algorithm 1 steps (2)-(3) without LayerNorm, LayerScale and
residual: QKV projection, router, per-head mode, concat, W_O.  With every
head routed to full it is standard multi-head attention.
global_block: Algorithm 1 in full: LN1, routed attention, LS1 + residual, LN2,
FFN (ratio 4, GELU), LS2 + residual.
"""
from __future__ import annotations

import numpy as np

from .modes import full_attention, linear_attention, mean_pooling, surrogate_attention
from .numerics import bf16_bits_to_f64, gelu, layer_norm, round_bf16
from .merge import destinations, key_metric, match, merge_tokens
from .position import qk_transform, token_positions
from .router import MODE_FULL, MODE_SURROGATE, attention_pool, routing_vector, saliency, select_mode

TAU_LOW = np.float32(0.01)     # §4.2 / App. B
TAU_HIGH = np.float32(0.20)
LN_EPS = 1e-6                  # not stated by the paper (reading)


def _identity(x):
    return np.asarray(x, np.float64)


def load_layer(w: dict) -> dict:
    """Decode one layer's stored parameters (bf16 bits / float32) to float64."""
    out = {}
    for k, v in w.items():
        v = np.asarray(v)
        out[k] = bf16_bits_to_f64(v) if v.dtype == np.uint16 else v.astype(np.float64)
    return out


def qkv_projection(Xt, lw, materialize=round_bf16, qk=None, tok_index=None):
    """Algorithm 1 step (2): (Q_h, K_h, V_h) <- QKV_h(X~).  A single linear map
    with bias whose 3D outputs are ordered (Q|K|V, head, channel); the returned
    array is [N, 3, H, d].  Positional information P (which the paper does not define)
    is off unless ``qk`` gives the reading of oracle.position: a dict with "q_norm" /
    "k_norm" ((gamma, beta) [d] or None), "eps", and "rope" (None or a dict with
    tokens_per_view, patch_start, grid_w, base); stored in bf16 after it.  tok_index: the
    token each row stands for (merged tokens), positions are that token's."""
    materialize = materialize or _identity
    N = Xt.shape[0]
    H = lw["r_W"].shape[0]
    qkv = (np.asarray(Xt, np.float64) @ lw["w_qkv"].T + lw["b_qkv"]).reshape(N, 3, H, -1)
    if qk is not None:
        rope = qk.get("rope")
        pos = None
        if rope is not None:
            toks = np.arange(N) if tok_index is None else np.asarray(tok_index)
            py, px = token_positions(int(toks.max()) + 1, rope["tokens_per_view"], rope["patch_start"],
                                     rope["grid_w"])
            pos = (py[toks], px[toks])
        base = None if rope is None else rope["base"]
        for h in range(H):
            qkv[:, 0, h] = qk_transform(qkv[:, 0, h], qk.get("q_norm"), qk.get("eps", 1e-6), pos, base)
            qkv[:, 1, h] = qk_transform(qkv[:, 1, h], qk.get("k_norm"), qk.get("eps", 1e-6), pos, base)
    return materialize(qkv)


# Ablation variants of §5 (component ablation and compute-mode ablation).  Two-branch
# routing (mean and full only) is tau_low == tau_high with the ordinary routing rule.
VARIANTS = ("mean_qpool", "mean_context", "no_residual", "linear_attention")


def head_router(Q_h, K_h, lw, h, beta=None, mean_qpool=False):
    """§4.1 for head h: (alpha, q_pool, r_h, s_h)."""
    d = Q_h.shape[1]
    alpha, q_pool = attention_pool(Q_h, lw["r_W"][h], lw["r_U"][h], lw["r_w"][h],
                                   lw["r_bW"][h], lw["r_bU"][h], mean_pool=mean_qpool)
    b = lw["r_beta"][h] if beta is None else beta
    r = routing_vector(q_pool, K_h, b / np.sqrt(d))
    return alpha, q_pool, r, saliency(r)


def moh_attention(X, lw, force_modes=None, rows=None, materialize=round_bf16,
                  tau_low=TAU_LOW, tau_high=TAU_HIGH, variant=(), qk=None, tok_index=None):
    """Routed multi-head attention of one layer (Algorithm 1 steps 2-3 up to W_O).

    X [N, D] float64 (the block passes LN1(X)); lw from load_layer.
    force_modes [H] replaces the routing decision only (the router still runs;
    surrogate heads still use its r_h).  ``rows`` restricts the per-token
    outputs to a subset of query rows (all rows when None); router statistics
    always use every token.  ``variant``: names from VARIANTS (§5 ablations).
    """
    variant = set(variant)
    assert variant <= set(VARIANTS), variant
    mat = materialize or _identity
    X = np.asarray(X, np.float64)
    N = X.shape[0]
    qkv = qkv_projection(X, lw, materialize, qk=qk, tok_index=tok_index)
    H, d = qkv.shape[2], qkv.shape[3]
    idx = np.arange(N) if rows is None else np.asarray(rows)
    res = {"qkv": qkv, "q_pool": np.zeros((H, d)), "s": np.zeros(H), "ctx": np.zeros((H, d)),
           "mean_v": np.zeros((H, d)), "alpha": [], "r": [], "rows": idx}
    Y = np.zeros((len(idx), H, d))
    natural = np.zeros(H, np.int32)
    modes = np.zeros(H, np.int32)
    for h in range(H):
        Q_h, K_h, V_h = qkv[:, 0, h], qkv[:, 1, h], qkv[:, 2, h]
        alpha, q_pool, r, s = head_router(Q_h, K_h, lw, h, mean_qpool="mean_qpool" in variant)
        res["alpha"].append(alpha)
        res["r"].append(r)
        res["q_pool"][h] = q_pool
        res["s"][h] = s
        natural[h] = select_mode(s, tau_low, tau_high)
        modes[h] = natural[h] if force_modes is None else int(force_modes[h])
        res["ctx"][h] = r @ V_h
        res["mean_v"][h] = V_h.sum(axis=0) / N
        if modes[h] == MODE_FULL:
            Y[:, h] = full_attention(Q_h, K_h, V_h, rows=idx)
        elif modes[h] == MODE_SURROGATE and "linear_attention" in variant:
            Y[:, h] = linear_attention(Q_h, K_h, V_h, rows=idx)
        elif modes[h] == MODE_SURROGATE:
            mg = (lw["s_g1_w"][h], lw["s_g1_b"][h], lw["s_g2_w"][h], lw["s_g2_b"][h])
            md = (lw["s_d1_w"][h], lw["s_d1_b"][h], lw["s_d2_w"][h], lw["s_d2_b"][h])
            Y[:, h], _ = surrogate_attention(V_h, r, mg, md, rows=idx,
                                             mean_context="mean_context" in variant,
                                             residual="no_residual" not in variant)
        else:
            Y[:, h], _ = mean_pooling(V_h, n_rows=len(idx))
    res["natural_modes"] = natural
    res["modes"] = modes
    res["Y"] = mat(Y.reshape(len(idx), H * d))          # Concat(Y_1..Y_H)
    res["out"] = mat(res["Y"] @ lw["w_o"].T + lw["b_o"])  # Y W_O (+ bias)
    return res


def global_block(X, lw, force_modes=None, materialize=round_bf16, eps=LN_EPS,
                 tau_low=TAU_LOW, tau_high=TAU_HIGH, variant=(), qk=None, merge=None, assign=None):
    """Algorithm 1 (VGGT-Prime global aggregator block), all rows.

    (1) X~ = LN1(X); (2) routed attention -> Y; (3) A = LS1(Y W_O),
    X_attn = X + A; (4) Z~ = LN2(X_attn), F = LS2(FFN(Z~)), X' = X_attn + F.
    FFN = Linear(D -> 4D) -> GELU -> Linear(4D -> D).  Returns (X', info).

    Storage points (materialize, bf16): QKV, Y, Z~, the FFN hidden layer and the residual
    stream X_attn, X'.  The LN1 output X~ is not stored: the block feeds it straight into
    the QKV projection, or, with merging, into the key metric and the merged tokens.

    merge: token merging around the attention (oracle.merge; a dict with stride,
    tokens_per_view, patch_start): X~ is merged (the merged tokens are stored), the routed
    attention and W_O (+ b_O, stored) run on the merged tokens, and every token adds LS1 times
    its merged token's output.  assign: the merged row of every token to use instead of the
    oracle's matching (the library's choice, for parity downstream of a near-tie)."""
    mat = materialize or _identity
    X = np.asarray(X, np.float64)
    Xt = layer_norm(X, lw["ln1_g"], lw["ln1_b"], eps)
    merged = None
    if merge is not None:
        row_of, dst_tok = destinations(X.shape[0], merge["tokens_per_view"], merge["patch_start"],
                                       merge["stride"])
        own, scores = match(key_metric(Xt, lw), row_of, dst_tok)
        asg = own if assign is None else np.asarray(assign)
        Xm = mat(merge_tokens(Xt, asg, len(dst_tok)))
        att = moh_attention(Xm, lw, force_modes=force_modes, materialize=materialize, tau_low=tau_low,
                            tau_high=tau_high, variant=variant, qk=qk, tok_index=dst_tok)
        A = att["out"][asg] * lw["ls1"]
        merged = {"assign": own, "scores": scores, "dst_tok": dst_tok}
    else:
        att = moh_attention(Xt, lw, force_modes=force_modes, materialize=materialize,
                            tau_low=tau_low, tau_high=tau_high, variant=variant, qk=qk)
        A = (att["Y"] @ lw["w_o"].T + lw["b_o"]) * lw["ls1"]
    X_attn = mat(X + A)
    Zt = mat(layer_norm(X_attn, lw["ln2_g"], lw["ln2_b"], eps))
    Hd = mat(gelu(Zt @ lw["w_fc1"].T + lw["b_fc1"]))
    F = (Hd @ lw["w_fc2"].T + lw["b_fc2"]) * lw["ls2"]
    X_next = mat(X_attn + F)
    return X_next, {"modes": att["modes"], "natural_modes": att["natural_modes"],
                    "s": att["s"], "X_attn": X_attn, "qkv": att["qkv"], "merge": merged}


def global_stack(X, layers, force_modes=None, materialize=round_bf16, eps=LN_EPS, variant=(),
                 qk=None, merge=None, assign=None):
    """Algorithm 1 applied layer after layer.  force_modes: [n_layers, H] or None;
    qk, merge, assign: per-layer lists of global_block's options, or None.
    Returns (X_out, list of per-layer info)."""
    infos = []
    for l, lw in enumerate(layers):
        fm = None if force_modes is None else force_modes[l]
        X, info = global_block(X, lw, force_modes=fm, materialize=materialize, eps=eps,
                               variant=variant, qk=None if qk is None else qk[l],
                               merge=None if merge is None else merge[l],
                               assign=None if assign is None else assign[l])
        infos.append(info)
    return X, infos
