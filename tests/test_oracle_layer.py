"""Pins of the oracle's layer and block (Algorithm 1) against textbook transformer
components from torch (CPU, float64), plus invariants and the paper's constants."""
import json
import os

import numpy as np
import pytest
import torch

import oracle
import synth
from oracle import MODE_FULL, MODE_MEAN, MODE_SURROGATE

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")
D, H, d, L = 256, 4, 64, 64


def _weights(seed, block=False, **kw):
    w = synth.make_layer_weights(synth.rng(seed), D=D, H=H, d=d, L=L, block=block,
                                 bias_std=0.1, norm_jitter=0.2 if block else 0.0, **kw)
    return oracle.load_layer(w)


def _torch_mha(X, lw):
    t = lambda a: torch.from_numpy(np.ascontiguousarray(a))
    out, _ = torch.nn.functional.multi_head_attention_forward(
        t(X)[:, None, :], t(X)[:, None, :], t(X)[:, None, :], D, H,
        t(lw["w_qkv"]), t(lw["b_qkv"]), None, None, False, 0.0,
        t(lw["w_o"]), t(lw["b_o"]), training=False, need_weights=False)
    return out[:, 0, :].numpy()


def test_all_full_layer_is_standard_multihead_attention():
    lw = _weights(0)
    X = np.random.default_rng(0).standard_normal((150, D))
    res = oracle.moh_attention(X, lw, force_modes=np.full(H, MODE_FULL), materialize=None)
    np.testing.assert_allclose(res["out"], _torch_mha(X, lw), rtol=1e-10, atol=1e-12)


def test_all_full_block_is_standard_prenorm_block():
    lw = _weights(1, block=True)
    X = np.random.default_rng(1).standard_normal((120, D))
    out, _ = oracle.global_block(X, lw, force_modes=np.full(H, MODE_FULL), materialize=None)
    t = lambda a: torch.from_numpy(np.ascontiguousarray(a))
    x = t(X)
    ln1 = torch.nn.functional.layer_norm(x, (D,), t(lw["ln1_g"]), t(lw["ln1_b"]), 1e-6)
    x_attn = x + t(lw["ls1"]) * torch.from_numpy(_torch_mha(ln1.numpy(), lw))
    ln2 = torch.nn.functional.layer_norm(x_attn, (D,), t(lw["ln2_g"]), t(lw["ln2_b"]), 1e-6)
    hid = torch.nn.functional.gelu(torch.nn.functional.linear(ln2, t(lw["w_fc1"]), t(lw["b_fc1"])))
    ref = x_attn + t(lw["ls2"]) * torch.nn.functional.linear(hid, t(lw["w_fc2"]), t(lw["b_fc2"]))
    np.testing.assert_allclose(out, ref.numpy(), rtol=1e-10, atol=1e-11)


def test_mean_and_surrogate_heads_use_their_operators():
    lw = _weights(2)
    X = np.random.default_rng(2).standard_normal((90, D))
    fm = np.array([MODE_MEAN, MODE_SURROGATE, MODE_FULL, MODE_MEAN])
    res = oracle.moh_attention(X, lw, force_modes=fm, materialize=None)
    qkv = res["qkv"]
    Y = res["Y"].reshape(90, H, d)
    np.testing.assert_allclose(Y[:, 0], np.tile(qkv[:, 2, 0].mean(0), (90, 1)), rtol=1e-12)
    np.testing.assert_allclose(Y[:, 3], np.tile(qkv[:, 2, 3].mean(0), (90, 1)), rtol=1e-12)
    np.testing.assert_allclose(Y[:, 2], oracle.full_attention(qkv[:, 0, 2], qkv[:, 1, 2], qkv[:, 2, 2]), rtol=1e-12)
    # The surrogate head's context is r_h V_h with the router's own r_h.
    np.testing.assert_allclose(res["ctx"][1], res["r"][1] @ qkv[:, 2, 1], rtol=1e-12)
    assert np.all(res["natural_modes"] >= 0)


def test_view_permutation_permutes_outputs():
    S, P = 5, 37
    lw = _weights(3)
    lw["r_beta"] = np.array([1.0, 80.0, 600.0, 8000.0])
    X = np.random.default_rng(3).standard_normal((S * P, D))
    perm = np.array([3, 0, 4, 1, 2])
    Xp = X.reshape(S, P, D)[perm].reshape(S * P, D)
    tok = (np.arange(S * P).reshape(S, P)[perm]).reshape(-1)
    a = oracle.moh_attention(X, lw, materialize=None)
    b = oracle.moh_attention(Xp, lw, materialize=None)
    np.testing.assert_allclose(b["s"], a["s"], rtol=1e-10)
    np.testing.assert_array_equal(b["modes"], a["modes"])
    np.testing.assert_allclose(b["out"], a["out"][tok], rtol=1e-10, atol=1e-12)
    np.testing.assert_allclose(b["ctx"], a["ctx"], rtol=1e-10, atol=1e-13)
    # The same holds for any token permutation and for every forced mode.
    for m in (MODE_MEAN, MODE_SURROGATE, MODE_FULL):
        pt = np.random.default_rng(m).permutation(S * P)
        fa = oracle.moh_attention(X, lw, force_modes=np.full(H, m), materialize=None)
        fb = oracle.moh_attention(X[pt], lw, force_modes=np.full(H, m), materialize=None)
        np.testing.assert_allclose(fb["out"], fa["out"][pt], rtol=1e-10, atol=1e-12)


def test_materialized_rounding_points_are_bf16():
    lw = _weights(4, block=True)
    X = oracle.round_bf16(np.random.default_rng(4).standard_normal((60, D)))
    out, info = oracle.global_block(X, lw)
    for arr in (out, info["X_attn"]):
        np.testing.assert_array_equal(oracle.round_bf16(arr), arr)


def test_stack_applies_blocks_in_order():
    lws = [_weights(10 + i, block=True) for i in range(3)]
    X = np.random.default_rng(5).standard_normal((40, D))
    fm = np.array([[MODE_FULL] * H, [MODE_MEAN] * H, [MODE_SURROGATE] * H])
    out, infos = oracle.global_stack(X, lws, force_modes=fm, materialize=None)
    x = X
    for l in range(3):
        x, _ = oracle.global_block(x, lws[l], force_modes=fm[l], materialize=None)
    np.testing.assert_array_equal(out, x)
    assert [list(i["modes"]) for i in infos] == [list(f) for f in fm]


def test_routing_distribution_constants():
    c = json.load(open(os.path.join(GOLDEN, "paper_constants.json")))["routing_distribution_percent"]
    rows = np.array(list(c["rows"].values()))
    np.testing.assert_allclose(rows.sum(1), 100.0, atol=0.15)
    avg = np.array(c["average"])
    assert abs(avg.sum() - 100.0) < 1e-9
    # The printed average is close to, but not exactly, the unweighted row mean.
    np.testing.assert_allclose(rows.mean(0), avg, atol=0.35)
    for k, v in zip(("mean", "surrogate", "full"), avg):
        assert abs(synth.PAPER_MIX[k] - v / 100) < 1e-12
    m = synth.paper_mix_modes(24, 16)
    assert (m == MODE_FULL).sum() == round(0.078 * 384)
    assert (m == MODE_MEAN).sum() == round(0.5 * 384)
