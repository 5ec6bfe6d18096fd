"""Full-size parity of the long-sequence stack's workload: S = 100 views at 518 px
(137,400 tokens), block 0 of the 24-block stack with its routes from the trained router's
average mix (2 full, 6 surrogate and 8 mean heads), against the float64 oracle.

At this size the router splits each head's pooling and key sweeps over 64 CTAs, and the
full-attention kernel splits the last round of its work groups along the keys, so these
tests check the split plans at the size the headline throughput is measured on:
  - the router (§4.1, §4.2) and every head mode (Algorithm 1 step 2, §4.3) on the oracle's
    own bf16 QKV bytes (identical inputs): s, routes, q_pool, C_h, mean of V, r_h on sampled
    tokens, and the head outputs Y on ~1,000 sampled rows that span the split groups;
  - the whole block (Algorithm 1) through vp_global_stack, with the paper-mix routes and
    with natural routing where two routers are steered into the full and surrogate bands:
    routes, saliencies and the block output on the sampled rows.
The oracle computes every router statistic over all 137,400 tokens and the per-token steps
on the sampled rows only (rows are independent given the router's outputs)."""
import numpy as np
import pytest
import torch

import oracle
import synth
from tests.helpers import BF16_STEP, TARGET_FULL, TARGET_SURROGATE, calibrate_beta, compare

pytestmark = pytest.mark.gpu

vpb = pytest.importorskip("paper_2609_23733_gb300.binding")

WL = synth.WORKLOADS["s100_stack"]
N, H = WL.N, synth.N_HEADS
EPS = 1e-6


@pytest.fixture(scope="module", autouse=True)
def _gpu():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    vpb.lib()


def _f64(t):
    return t.detach().float().cpu().numpy().astype(np.float64)


def _sample_rows(n_full):
    """~1,000 rows: the ends, the first rows of the last (split) round of full-attention
    groups on 152 SMs, and a seeded spread.  Groups are three 128-row tiles, head-major."""
    tiles = -(-N // 128)
    groups_per_head = -(-tiles // 3)
    tail_group = (n_full * groups_per_head // 152) * 152  # first group of the last round
    tail_row = (tail_group % groups_per_head) * 384
    parts = [np.arange(0, 64), np.arange(N - 64, N), np.arange(tail_row, min(N, tail_row + 96)),
             np.random.default_rng(100).choice(N, 800, replace=False)]
    return np.unique(np.concatenate(parts))


def _mlps(lw, h):
    return ((lw["s_g1_w"][h], lw["s_g1_b"][h], lw["s_g2_w"][h], lw["s_g2_b"][h]),
            (lw["s_d1_w"][h], lw["s_d1_b"][h], lw["s_d2_w"][h], lw["s_d2_b"][h]))


def _oracle_heads(qkv, lw, modes, rows):
    """Router statistics of every head over all tokens, and Y on ``rows`` (float64)."""
    out = {"s": np.zeros(H), "q_pool": np.zeros((H, 64)), "ctx": np.zeros((H, 64)),
           "mean_v": np.zeros((H, 64)), "r": np.zeros((H, N)), "Y": np.zeros((len(rows), H, 64))}
    for h in range(H):
        Q, K, V = qkv[:, 0, h], qkv[:, 1, h], qkv[:, 2, h]
        _, q_pool, r, s = oracle.layer.head_router(Q, K, lw, h)
        out["s"][h], out["q_pool"][h], out["r"][h] = s, q_pool, r
        out["ctx"][h], out["mean_v"][h] = r @ V, V.sum(0) / N
        if modes[h] == synth.MODE_FULL:
            out["Y"][:, h] = oracle.full_attention(Q, K, V, rows=rows)
        elif modes[h] == synth.MODE_SURROGATE:
            out["Y"][:, h], _ = oracle.surrogate_attention(V, r, *_mlps(lw, h), rows=rows)
        else:
            out["Y"][:, h], _ = oracle.mean_pooling(V, n_rows=len(rows))
    return out


def _block_rows(X_rows, Y_rows, lw):
    """Algorithm 1 steps (3)-(4) for the sampled rows, given their head outputs."""
    Y = oracle.round_bf16(Y_rows.reshape(len(Y_rows), -1))
    Xa = oracle.round_bf16(X_rows + (Y @ lw["w_o"].T + lw["b_o"]) * lw["ls1"])
    Zt = oracle.round_bf16(oracle.layer_norm(Xa, lw["ln2_g"], lw["ln2_b"], EPS))
    Hd = oracle.round_bf16(oracle.gelu(Zt @ lw["w_fc1"].T + lw["b_fc1"]))
    return oracle.round_bf16(Xa + (Hd @ lw["w_fc2"].T + lw["b_fc2"]) * lw["ls2"])


@pytest.fixture(scope="module")
def _case():
    w = synth.make_stack_weights(WL.seed, 1)[0]  # block 0 of the stack (same draws as 24 blocks)
    routes = synth.paper_mix_modes(WL.layers)[0]
    x_bits = synth.make_tokens(WL.seed, N)
    lw = oracle.load_layer(w)
    X = oracle.bf16_bits_to_f64(x_bits)
    qkv = oracle.qkv_projection(oracle.layer_norm(X, lw["ln1_g"], lw["ln1_b"], EPS), lw)
    rows = _sample_rows(int((routes == synth.MODE_FULL).sum()))
    want = _oracle_heads(qkv, lw, routes, rows)
    return {"w": w, "lw": lw, "routes": routes, "x_bits": x_bits, "X_rows": X[rows], "qkv": qkv,
            "rows": rows, "want": want}


def test_s100_router_and_heads_on_identical_qkv(_case):
    qkv, w, routes, rows, want = _case["qkv"], _case["w"], _case["routes"], _case["rows"], _case["want"]
    assert sorted(np.bincount(routes, minlength=3).tolist()) == [2, 6, 8]
    qkv_dev = vpb.bf16_from_bits(synth.f32_to_bf16_bits(qkv.reshape(N, -1).astype(np.float32)))
    dw = vpb.to_device(w)
    dm = vpb.dims(N, H)
    ws = vpb.workspace(dm, vpb.VP_WS_ROUTER)
    s = torch.zeros(H, device="cuda")
    modes = torch.full((H,), -1, dtype=torch.int32, device="cuda")
    q_pool, ctx, mean_v = (torch.zeros(H, 64, device="cuda") for _ in range(3))
    r = torch.zeros(H, N, device="cuda")
    vpb.vp_router(dm, qkv_dev, vpb.router_weights(dw), None, s, modes, q_pool, ctx, mean_v, r, ws)
    torch.cuda.synchronize()
    assert vpb.vp_read_device_error(ws) == 0
    np.testing.assert_allclose(_f64(s), want["s"], rtol=2e-4, atol=1e-9)
    want_modes = [oracle.select_mode(v) for v in want["s"]]  # untrained routers: every head mean
    np.testing.assert_array_equal(modes.cpu().numpy(), want_modes)
    np.testing.assert_allclose(_f64(q_pool), want["q_pool"], rtol=2e-3, atol=2e-4)
    np.testing.assert_allclose(_f64(ctx), want["ctx"], rtol=2e-3, atol=2e-4)
    np.testing.assert_allclose(_f64(mean_v), want["mean_v"], rtol=1e-4, atol=1e-5)
    toks = np.unique(np.concatenate([rows, np.random.default_rng(101).choice(N, 4000, replace=False)]))
    got_r = _f64(r)
    np.testing.assert_allclose(got_r[:, toks], want["r"][:, toks], rtol=2e-3, atol=1e-10)
    np.testing.assert_allclose(got_r.sum(1), 1.0, atol=1e-4)
    # Head outputs with the paper-mix routes (bins and router outputs from the oracle).
    ids, off, _ = oracle.bin_heads(routes, N)
    y = torch.full((N, H * 64), float("nan"), dtype=torch.bfloat16, device="cuda")
    vpb.vp_head_attention(dm, qkv_dev, torch.tensor(ids, device="cuda"), torch.tensor(off, device="cuda"),
                          torch.tensor(want["ctx"], dtype=torch.float32, device="cuda"),
                          torch.tensor(want["mean_v"], dtype=torch.float32, device="cuda"),
                          vpb.surrogate_weights(dw), y, ws)
    torch.cuda.synchronize()
    assert vpb.vp_read_device_error(ws) == 0
    got_y = _f64(y).reshape(N, H, 64)
    assert np.all(np.isfinite(got_y))  # every row of every head was written
    got_y = got_y[rows]
    for h in range(H):
        compare(got_y[:, h], oracle.round_bf16(want["Y"][:, h]), what=f"head {h} mode {routes[h]}")


def _run_block(x_bits, w, force):
    dm = vpb.dims(N, H)
    dw = vpb.to_device(w)
    ws = vpb.workspace(dm, vpb.VP_WS_STACK)
    x = vpb.bf16_from_bits(x_bits)
    modes = torch.full((1, H), -1, dtype=torch.int32, device="cuda")
    s = torch.zeros(1, H, device="cuda")
    fm = None if force is None else torch.tensor(np.asarray(force, np.int32)[None], device="cuda")
    vpb.vp_global_stack(dm, x, [vpb.layer_weights(dw)], fm, modes, s, EPS, ws)
    torch.cuda.synchronize()
    assert vpb.vp_read_device_error(ws) == 0
    return _f64(x), modes.cpu().numpy()[0], s.cpu().numpy()[0].astype(np.float64)


def test_s100_block0_paper_mix(_case):
    got, modes, s = _run_block(_case["x_bits"], _case["w"], _case["routes"])
    np.testing.assert_array_equal(modes, _case["routes"])
    # the block's own QKV (LN1 folded into the projection) rounds independently of the oracle's
    np.testing.assert_allclose(s, _case["want"]["s"], rtol=5e-3)
    rows = _case["rows"]
    want = _block_rows(_case["X_rows"], _case["want"]["Y"], _case["lw"])
    compare(got[rows], want, rel=BF16_STEP, what="S=100 block 0, paper-mix routes (sampled rows)")


def test_s100_block0_natural_routing_with_steered_heads():
    """Natural routing at full size: the routers of heads 0 and 1 are steered (per-head beta,
    bisected on the oracle) to saliency 0.5 and sqrt(0.01 * 0.2), the middles of the full and
    surrogate bands; the other 14 stay untrained (mean)."""
    w = synth.make_layer_weights(synth.rng(WL.seed), block=True)
    x_bits = synth.make_tokens(WL.seed, N)
    lw = oracle.load_layer(w)
    X = oracle.bf16_bits_to_f64(x_bits)
    qkv = oracle.qkv_projection(oracle.layer_norm(X, lw["ln1_g"], lw["ln1_b"], EPS), lw)
    for h, target in ((0, TARGET_FULL), (1, TARGET_SURROGATE)):
        w["r_beta"][h] = calibrate_beta(qkv, lw, h, target)
    lw["r_beta"] = w["r_beta"].astype(np.float64)
    rows = _sample_rows(1)
    routes = np.array([synth.MODE_FULL, synth.MODE_SURROGATE] + [synth.MODE_MEAN] * (H - 2), np.int32)
    want = _oracle_heads(qkv, lw, routes, rows)
    np.testing.assert_array_equal([oracle.select_mode(v) for v in want["s"]], routes)
    # whole-block runs round QKV on each side: the routes are compared 5 % away from a threshold
    assert abs(want["s"][0] - 0.2) > 0.05 * 0.2 and abs(want["s"][1] - 0.01) > 0.05 * 0.01
    got, modes, s = _run_block(x_bits, w, None)
    np.testing.assert_array_equal(modes, routes)
    np.testing.assert_allclose(s, want["s"], rtol=2e-2)
    compare(got[rows], _block_rows(X[rows], want["Y"], lw), rel=BF16_STEP,
            what="S=100 block 0, natural routing (sampled rows)")
