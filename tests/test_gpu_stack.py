"""GPU parity of Algorithm 1's block stack (vp_global_stack) and the routing-mix sweep at
full size (S = 64 views, 87,936 tokens) against the float64 oracle.

Stack outputs are the residual stream, stored in bf16 after every block (LayerScale 1
gives it magnitude > 1), so besides the absolute bar they allow one bf16 step relative to
the value per block boundary that rounding can cross, and deep stacks use a per-block error
budget times the depth (see test_stack_24_blocks_s4_natural_routing)."""
import numpy as np
import pytest
import torch

import oracle
import synth
from tests.helpers import BF16_STEP, compare

pytestmark = pytest.mark.gpu

vpb = pytest.importorskip("paper_2609_23733_gb300.binding")


@pytest.fixture(scope="module", autouse=True)
def _gpu():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    vpb.lib()


def _f64(t):
    return t.detach().float().cpu().numpy().astype(np.float64)


def _run_stack(x_bits, ws_host, N, force=None, H=16):
    dm = vpb.dims(N, H)
    dws = [vpb.to_device(w) for w in ws_host]
    layers = [vpb.layer_weights(w) for w in dws]
    ws = vpb.workspace(dm, vpb.VP_WS_STACK)
    x = vpb.bf16_from_bits(x_bits)
    L = len(ws_host)
    modes = torch.full((L, H), -1, dtype=torch.int32, device="cuda")
    s = torch.zeros(L, H, device="cuda")
    s_attn = torch.full((L, H), float("nan"), device="cuda")
    fm = None if force is None else torch.tensor(np.asarray(force, np.int32), device="cuda")
    vpb.vp_global_stack(dm, x, layers, fm, modes, s, 1e-6, ws, s_attn_out=s_attn)
    torch.cuda.synchronize()
    assert vpb.vp_read_device_error(ws) == 0
    _run_stack.s_attn = s_attn.cpu().numpy().astype(np.float64)
    return _f64(x), modes.cpu().numpy(), s.cpu().numpy()


def test_stack_host_buffers_equal_the_device_path():
    """vp_global_stack_host (tokens in page-locked host memory, copied by the library's own
    kernel both ways) gives the bits of vp_global_stack on a device copy of the tokens, in
    place (x_out = x_in) and into a second buffer; unpinned host memory is refused."""
    N, L, H = 1000, 2, 16
    g = synth.rng(41)
    wts = [synth.make_layer_weights(g, block=True, bias_std=0.05) for _ in range(L)]
    x_bits = synth.make_tokens(41, N)
    force = np.array([synth.forced_mix(H, f) for f in (0.25, 0.0)])
    dm = vpb.dims(N, H)
    dws = [vpb.to_device(w) for w in wts]
    layers = [vpb.layer_weights(w) for w in dws]
    ws = vpb.workspace(dm, vpb.VP_WS_STACK)
    fm = torch.tensor(force, device="cuda")
    modes = torch.zeros(L, H, dtype=torch.int32, device="cuda")
    s = torch.zeros(L, H, device="cuda")
    x = vpb.bf16_from_bits(x_bits)
    vpb.vp_global_stack(dm, x, layers, fm, modes, s, 1e-6, ws)
    torch.cuda.synchronize()
    want = x.cpu()
    host_in = vpb.bf16_from_bits(x_bits).cpu().pin_memory()
    host_out = torch.zeros_like(host_in).pin_memory()
    x_dev = torch.empty(N, H * 64, dtype=torch.bfloat16, device="cuda")
    for out in (host_out, host_in):  # into a second buffer, then in place
        vpb.vp_global_stack_host(dm, host_in, out, x_dev, layers, fm, modes, s, 1e-6, ws)
        torch.cuda.synchronize()
        assert vpb.vp_read_device_error(ws) == 0
        assert torch.equal(out, want)
    pageable = vpb.bf16_from_bits(x_bits).cpu()
    with pytest.raises(vpb.VPError) as e:
        vpb.vp_global_stack_host(dm, pageable, host_out, x_dev, layers, fm, modes, s, 1e-6, ws)
    assert e.value.status == 1  # VP_ERR_INVALID_ARG: not page-locked


def test_stack_three_blocks_all_modes():
    N, L = 600, 3
    g = synth.rng(5)
    wts = [synth.make_layer_weights(g, block=True, bias_std=0.05, norm_jitter=0.1) for _ in range(L)]
    for w in wts:
        w["ls1"] = (0.5 * w["ls1"]).astype(np.float32)
        w["ls2"] = (0.5 * w["ls2"]).astype(np.float32)
    x_bits = synth.make_tokens(5, N)
    force = np.array([synth.forced_mix(16, f) for f in (0.25, 0.5, 1.0)])
    got, modes, s = _run_stack(x_bits, wts, N, force)
    want, infos = oracle.global_stack(oracle.bf16_bits_to_f64(x_bits), [oracle.load_layer(w) for w in wts],
                                      force_modes=force)
    np.testing.assert_array_equal(modes, force)
    np.testing.assert_allclose(s[0], infos[0]["s"], rtol=5e-3)
    compare(got, want, rel=L * BF16_STEP, what="3-block stack")
    # MaxAttn saliency per block for the full heads (0 for the others); later blocks see the
    # residual stream after the earlier blocks' independent roundings, hence 2 %
    for l in range(L):
        for h in range(16):
            got_s = _run_stack.s_attn[l, h]
            if force[l][h] == synth.MODE_FULL:
                q = infos[l]["qkv"]
                ref = oracle.max_attention_saliency(q[:, 0, h], q[:, 1, h])
                assert abs(got_s - ref) <= 2e-2 * ref, (l, h, got_s, ref)
            else:
                assert got_s == 0.0, (l, h, got_s)


def test_stack_repeated_runs_are_bit_identical():
    """Two runs of a 3-block stack at 6,000 tokens (every route, several tiles per pooling CTA)
    on the same tokens give the same bits: every reduction in the library has a fixed order
    (token merging is not part of this, since a merged token sums its members in fill order)."""
    N, L = 6000, 3
    g = synth.rng(7)
    wts = [synth.make_layer_weights(g, block=True, bias_std=0.05, norm_jitter=0.1) for _ in range(L)]
    x_bits = synth.make_tokens(7, N)
    force = np.array([synth.forced_mix(16, f) for f in (0.25, 0.5, 1.0)])
    a, ma, sa = _run_stack(x_bits, wts, N, force)
    sat_a = _run_stack.s_attn.copy()
    b, mb, sb = _run_stack(x_bits, wts, N, force)
    np.testing.assert_array_equal(a, b)
    np.testing.assert_array_equal(ma, mb)
    np.testing.assert_array_equal(sa, sb)
    np.testing.assert_array_equal(sat_a, _run_stack.s_attn)


def test_stack_24_blocks_s4_natural_routing():
    """24 blocks over S=4 views at 224 px (1,044 tokens): untrained routers route every
    head of every block to mean (saliency ~ 1/N)."""
    wl = synth.WORKLOADS["s4_layer"]
    N, L = wl.N, 24
    wts = synth.make_stack_weights(wl.seed, L)
    for w in wts:  # keep the residual stream O(1) over 24 blocks
        w["ls1"] = np.full_like(w["ls1"], 0.2)
        w["ls2"] = np.full_like(w["ls2"], 0.2)
    x_bits = synth.make_tokens(wl.seed, N)
    got, modes, s = _run_stack(x_bits, wts, N)
    want, infos = oracle.global_stack(oracle.bf16_bits_to_f64(x_bits), [oracle.load_layer(w) for w in wts])
    np.testing.assert_array_equal(modes, np.array([i["modes"] for i in infos]))
    assert np.all(modes == synth.MODE_MEAN)
    # Each block ends in bf16 storage of the residual stream; the two sides round independently
    # and the differences compound through later blocks, growing about linearly with depth
    # (measured on GB300: relative norm 2.8e-4 after one block, 6.5e-3 after 24).  The bar is
    # a per-block budget times the depth: relative norm 5e-4 and mean-abs 4e-4 per block.
    compare(got, want, max_abs=4e-2, mean_abs=L * 4e-4, rel=4 * BF16_STEP, what="24-block stack")
    err = np.linalg.norm(got - want) / np.linalg.norm(want)
    assert err < L * 5e-4, err


def _s32_case():
    wl = synth.WORKLOADS["s32_stack"]
    wts = synth.make_stack_weights(wl.seed, 24)
    for w in wts:  # keep the residual stream O(1) over 24 blocks
        w["ls1"] = np.full_like(w["ls1"], 0.2)
        w["ls2"] = np.full_like(w["ls2"], 0.2)
    return wl, wts, synth.make_tokens(wl.seed, wl.N)


@pytest.fixture(scope="module")
def _s32_oracle():
    """The oracle's 24 blocks over all 43,968 tokens: its input to every block (bf16 bits),
    its routes and saliencies, and its output."""
    wl, wts, x_bits = _s32_case()
    X = oracle.bf16_bits_to_f64(x_bits)
    inputs, infos = [], []
    for w in wts:
        inputs.append(synth.f32_to_bf16_bits(X.astype(np.float32)))  # exact: X holds bf16 values
        X, info = oracle.global_block(X, oracle.load_layer(w))
        infos.append({"modes": info["modes"], "s": info["s"]})
    return {"wl": wl, "wts": wts, "x_bits": x_bits, "inputs": inputs, "infos": infos, "out": X}


@pytest.mark.slow
@pytest.mark.parametrize("blk", [0, 11, 23])
def test_stack_s32_block_against_oracle(blk, _s32_oracle):
    """Full size S=32 (43,968 tokens): blocks 0, 11 and 23 of the 24-block stack, each run on
    the GPU from the oracle's own input to that block, against the oracle's output of that
    block on every row (routes exact; natural routing of the untrained routers)."""
    c = _s32_oracle
    N = c["wl"].N
    got, modes, s = _run_stack(c["inputs"][blk], c["wts"][blk:blk + 1], N)
    want = c["inputs"][blk + 1] if blk + 1 < 24 else synth.f32_to_bf16_bits(c["out"].astype(np.float32))
    np.testing.assert_array_equal(modes[0], c["infos"][blk]["modes"])
    np.testing.assert_allclose(s[0], c["infos"][blk]["s"], rtol=5e-3)
    compare(got, oracle.bf16_bits_to_f64(want), rel=BF16_STEP, what=f"S=32 block {blk}")


@pytest.mark.slow
def test_stack_s32_24_blocks_against_oracle(_s32_oracle):
    """The whole S=32 stack, 24 blocks on the GPU from the tokens, against the oracle's 24
    blocks: routes of every block exact, the output within the depth budget of
    test_stack_24_blocks_s4_natural_routing (each block's bf16 residual stream is rounded
    independently on the two sides, and the differences compound with depth)."""
    c = _s32_oracle
    L = 24
    got, modes, _ = _run_stack(c["x_bits"], c["wts"], c["wl"].N)
    np.testing.assert_array_equal(modes, np.array([i["modes"] for i in c["infos"]]))
    compare(got, c["out"], max_abs=4e-2, mean_abs=L * 4e-4, rel=4 * BF16_STEP, what="S=32, 24 blocks")
    err = np.linalg.norm(got - c["out"]) / np.linalg.norm(c["out"])
    assert err < L * 5e-4, err


def test_stack_s32_view_permutation():
    """The whole 24-block S=32 stack is equivariant under a permutation of the views (an
    invariant of the method at any size, checked GPU against GPU)."""
    wl, wts, x_bits = _s32_case()
    N, P, L = wl.N, wl.P, 24
    perm = np.random.default_rng(2).permutation(wl.views)
    xp_bits = x_bits.reshape(wl.views, P, -1)[perm].reshape(N, -1)
    out, modes, _ = _run_stack(x_bits, wts, N)
    outp, modesp, _ = _run_stack(xp_bits, wts, N)
    np.testing.assert_array_equal(modes, modesp)
    assert np.all(np.isfinite(out))
    ref = out.reshape(wl.views, P, -1)[perm].reshape(N, -1)
    # Exact in real arithmetic; numerically the router's and the mean heads' token sums run in
    # another order, and the differences compound like the stack's rounding (same budget).
    rel = np.linalg.norm(outp - ref) / np.linalg.norm(ref)
    assert rel < L * 5e-4, rel


@pytest.mark.parametrize("frac", [0.0, 0.25, 0.5, 1.0])
def test_mix_sweep_s64_sampled_rows(frac, _s64_case):
    """Single layer at S=64 views (87,936 tokens) with 0 / 25 / 50 / 100 % of the heads
    forced to full mode; every head checked on sampled rows against the oracle."""
    x_bits, w, lw, qkv, routers, rows = _s64_case
    N, H = qkv.shape[0], 16
    force = synth.forced_mix(H, frac)
    dm = vpb.dims(N, H)
    dw = vpb.to_device(w)
    ws = vpb.workspace(dm, vpb.VP_WS_LAYER)
    out = torch.zeros(N, H * 64, dtype=torch.bfloat16, device="cuda")
    y = torch.zeros(N, H * 64, dtype=torch.bfloat16, device="cuda")
    modes = torch.zeros(H, dtype=torch.int32, device="cuda")
    vpb.vp_moh_global_attention(dm, vpb.bf16_from_bits(x_bits), dw["w_qkv"], dw["b_qkv"], dw["w_o"], dw["b_o"],
                                vpb.router_weights(dw), vpb.surrogate_weights(dw),
                                torch.from_numpy(force).cuda(), out, None, y, None, modes, ws)
    torch.cuda.synchronize()
    assert vpb.vp_read_device_error(ws) == 0
    np.testing.assert_array_equal(modes.cpu().numpy(), force)
    Y = np.zeros((len(rows), H, 64))
    for h in range(H):
        Q, K, V = qkv[:, 0, h], qkv[:, 1, h], qkv[:, 2, h]
        r = routers[h]
        if force[h] == synth.MODE_FULL:
            Y[:, h] = oracle.full_attention(Q, K, V, rows=rows)
        elif force[h] == synth.MODE_SURROGATE:
            mg = (lw["s_g1_w"][h], lw["s_g1_b"][h], lw["s_g2_w"][h], lw["s_g2_b"][h])
            md = (lw["s_d1_w"][h], lw["s_d1_b"][h], lw["s_d2_w"][h], lw["s_d2_b"][h])
            Y[:, h], _ = oracle.surrogate_attention(V, r, mg, md, rows=rows)
        else:
            Y[:, h], _ = oracle.mean_pooling(V, n_rows=len(rows))
    Y = oracle.round_bf16(Y.reshape(len(rows), -1))
    compare(_f64(y)[rows], Y, what=f"Y at {frac:.0%} full")
    compare(_f64(out)[rows], oracle.round_bf16(Y @ lw["w_o"].T + lw["b_o"]), what=f"out at {frac:.0%} full")


@pytest.fixture(scope="module")
def _s64_case():
    wl = synth.WORKLOADS["s64_mix_sweep"]
    N = wl.N
    w = synth.make_layer_weights(synth.rng(wl.seed), bias_std=0.02)
    x_bits = synth.make_tokens(wl.seed, N)
    lw = oracle.load_layer(w)
    qkv = oracle.qkv_projection(oracle.bf16_bits_to_f64(x_bits), lw)
    routers = [oracle.layer.head_router(qkv[:, 0, h], qkv[:, 1, h], lw, h)[2] for h in range(16)]
    rows = np.unique(np.concatenate([np.arange(0, 130), np.arange(N - 130, N),
                                     np.random.default_rng(3).choice(N, 256, replace=False)]))
    return x_bits, w, lw, qkv, routers, rows
