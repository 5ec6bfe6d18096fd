"""GPU parity of §5's ablation variants (vp_dims.variant and tau_low == tau_high) against the
oracle: mean query pooling, mean-value context, no residual correction, linear attention
(phi = elu + 1) for the surrogate heads, and the two-branch router (mean and full only)."""
import numpy as np
import pytest
import torch

import oracle
import synth
from tests.helpers import calibrated_layer, compare, outside_guard

pytestmark = pytest.mark.gpu

vpb = pytest.importorskip("paper_2609_23733_gb300.binding")

FLAG = {"mean_qpool": 1, "mean_context": 2, "no_residual": 4, "linear_attention": 8}


@pytest.fixture(scope="module", autouse=True)
def _gpu():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    vpb.lib()


def _f64(t):
    return t.detach().float().cpu().numpy().astype(np.float64)


def _run_layer(x_bits, w, N, force=None, variant=(), tau=(0.01, 0.20), H=16):
    flags = sum(FLAG[v] for v in variant)
    dm = vpb.dims(N, H, tau_low=tau[0], tau_high=tau[1], variant=flags)
    dw = vpb.to_device(w)
    ws = vpb.workspace(dm, vpb.VP_WS_LAYER)
    out = torch.zeros(N, H * 64, dtype=torch.bfloat16, device="cuda")
    y = torch.zeros(N, H * 64, dtype=torch.bfloat16, device="cuda")
    s = torch.zeros(H, device="cuda")
    modes = torch.zeros(H, dtype=torch.int32, device="cuda")
    fm = None if force is None else torch.tensor(np.asarray(force, np.int32), device="cuda")
    vpb.vp_moh_global_attention(dm, vpb.bf16_from_bits(x_bits), dw["w_qkv"], dw["b_qkv"], dw["w_o"],
                                dw["b_o"], vpb.router_weights(dw), vpb.surrogate_weights(dw), fm, out,
                                None, y, s, modes, ws)
    torch.cuda.synchronize()
    assert vpb.vp_read_device_error(ws) == 0
    return _f64(out), _f64(y), s.cpu().numpy(), modes.cpu().numpy()


MIX = [2, 1, 0, 1] * 4  # 4 full, 8 surrogate, 4 mean


@pytest.mark.parametrize("variant", [("mean_qpool",), ("mean_context",), ("no_residual",),
                                     ("linear_attention",), ("mean_qpool", "mean_context"),
                                     ("mean_qpool", "linear_attention")])
def test_variant_layer_s4(variant):
    """S=4 views at 224 px (1,044 tokens), four full / eight surrogate / four mean heads."""
    wl = synth.WORKLOADS["s4_layer"]
    N = wl.N
    w = synth.make_layer_weights(synth.rng(wl.seed), bias_std=0.05)
    x_bits = synth.make_tokens(wl.seed, N)
    got, y, s, modes = _run_layer(x_bits, w, N, MIX, variant)
    want = oracle.moh_attention(oracle.bf16_bits_to_f64(x_bits), oracle.load_layer(w), force_modes=MIX,
                                variant=variant)
    np.testing.assert_array_equal(modes, MIX)
    np.testing.assert_allclose(s, want["s"], rtol=2e-3)
    compare(y, want["Y"], what=f"Y {variant}")
    compare(got, want["out"], what=f"out {variant}")


def test_mean_qpool_changes_only_the_router():
    """Mean pooling gives q_pool = mean query; every head's s and the natural routes follow."""
    wl = synth.WORKLOADS["s4_layer"]
    N = wl.N
    w = synth.make_layer_weights(synth.rng(wl.seed))
    x_bits = synth.make_tokens(wl.seed, N)
    _, _, s, modes = _run_layer(x_bits, w, N, None, ("mean_qpool",))
    want = oracle.moh_attention(oracle.bf16_bits_to_f64(x_bits), oracle.load_layer(w), variant=("mean_qpool",))
    np.testing.assert_allclose(s, want["s"], rtol=2e-3)
    np.testing.assert_array_equal(modes, want["modes"])
    base = oracle.moh_attention(oracle.bf16_bits_to_f64(x_bits), oracle.load_layer(w))
    assert not np.allclose(want["s"], base["s"], rtol=1e-3)  # the ablation is visible in s


def test_two_branch_router():
    """tau_low == tau_high = 0.1: heads steered to s = 0.5 run full, heads steered into the
    old surrogate band (s = 0.045) and unsteered heads (s ~ 1/N) run mean; no surrogate band."""
    wl = synth.WORKLOADS["s4_layer"]
    N = wl.N
    mix = [2, 1, 0, 1, 1, 2, 0, 0, 1, 0, 2, 1, 0, 1, 0, 0]
    x_bits, w, lw = calibrated_layer(wl.seed, N, mix)
    tau = 0.1
    got, y, s, modes = _run_layer(x_bits, w, N, None, (), (tau, tau))
    want = oracle.moh_attention(oracle.bf16_bits_to_f64(x_bits), lw, tau_low=np.float32(tau),
                                tau_high=np.float32(tau))
    assert np.all(outside_guard(want["s"], tau_low=tau, tau_high=tau, guard=0.05))
    np.testing.assert_array_equal(modes, want["modes"])
    np.testing.assert_array_equal(modes, [2 if m == 2 else 0 for m in mix])
    compare(got, want["out"], what="two-branch out")


@pytest.mark.parametrize("N", [1, 63, 64, 129, 2000, 9999])
def test_linear_attention_heads(N):
    """vp_head_attention with the linear-attention variant: every surrogate head against the
    oracle's definition, at sizes with ragged state tiles and several state splits."""
    H = 4
    g = np.random.default_rng(N)
    qkv = (g.standard_normal((N, 3, H, 64)) * 1.5).astype(np.float32)
    qkv[:, 2] += 0.3  # a nonzero mean, so that outputs are not all near 0
    qkv_bits = synth.f32_to_bf16_bits(qkv)
    q = oracle.bf16_bits_to_f64(qkv_bits).reshape(N, 3, H, 64)
    modes = np.array([1, 2, 1, 0], np.int32)
    ids_o, off_o, _ = oracle.bin_heads(modes, N)
    dm = vpb.dims(N, H, variant=FLAG["linear_attention"])
    w = vpb.to_device(synth.make_layer_weights(synth.rng(1), D=H * 64, H=H))
    ws = vpb.workspace(dm, vpb.VP_WS_ROUTER)
    y = torch.full((N, H * 64), float("nan"), dtype=torch.bfloat16, device="cuda")
    mv = torch.tensor(q[:, 2].mean(0), dtype=torch.float32, device="cuda")
    vpb.vp_head_attention(dm, vpb.bf16_from_bits(qkv_bits.reshape(N, -1)), torch.tensor(ids_o, device="cuda"),
                          torch.tensor(off_o, device="cuda"), torch.zeros(H, 64, device="cuda"), mv,
                          vpb.surrogate_weights(w), y, ws)
    torch.cuda.synchronize()
    assert vpb.vp_read_device_error(ws) == 0
    got = _f64(y).reshape(N, H, 64)
    for h in (0, 2):
        want = oracle.linear_attention(q[:, 0, h], q[:, 1, h], q[:, 2, h])
        compare(got[:, h], oracle.round_bf16(want), what=f"linear head {h}")
    compare(got[:, 1], oracle.round_bf16(oracle.full_attention(q[:, 0, 1], q[:, 1, 1], q[:, 2, 1])), what="full")
    compare(got[:, 3], oracle.round_bf16(np.tile(q[:, 2, 3].mean(0), (N, 1))), what="mean")


@pytest.mark.parametrize("N,H", [(50_000, 4), (137_400, 16)])
def test_linear_attention_heads_sampled_rows(N, H):
    """The linear-attention variant at sizes where every CTA of both kernels takes several
    token tiles (the 16-head, 137,400-token case is the S = 100 stack's head geometry): sampled
    rows of every linear head against the oracle's definition, and the mean head in full."""
    g = np.random.default_rng(N + H)
    # Standard normal x 1.5, drawn in bf16 by torch's seeded CPU generator (numpy's float32
    # draw and rounding take minutes at 422 M values).
    x = torch.randn(N, 3 * H * 64, generator=torch.Generator().manual_seed(N + H)) * 1.5
    bits = x.to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16).reshape(N, 3, H, 64)
    del x
    modes = np.ones(H, np.int32)
    modes[H - 1] = 0
    ids_o, off_o, _ = oracle.bin_heads(modes, N)
    dm = vpb.dims(N, H, variant=FLAG["linear_attention"])
    w = vpb.to_device(synth.make_layer_weights(synth.rng(1), D=H * 64, H=H))
    ws = vpb.workspace(dm, vpb.VP_WS_ROUTER)
    y = torch.full((N, H * 64), float("nan"), dtype=torch.bfloat16, device="cuda")
    v_last = oracle.bf16_bits_to_f64(bits[:, 2, H - 1])
    mv = torch.zeros(H, 64, dtype=torch.float32, device="cuda")
    mv[H - 1] = torch.tensor(v_last.mean(0), dtype=torch.float32)
    vpb.vp_head_attention(dm, vpb.bf16_from_bits(bits.reshape(N, -1)), torch.tensor(ids_o, device="cuda"),
                          torch.tensor(off_o, device="cuda"), torch.zeros(H, 64, device="cuda"), mv,
                          vpb.surrogate_weights(w), y, ws)
    torch.cuda.synchronize()
    assert vpb.vp_read_device_error(ws) == 0
    got = y.float().cpu().numpy().reshape(N, H, 64)
    edges = [0, 1, 127, 128, 129, N // 2, N - 129, N - 128, N - 1]
    for h in range(H - 1):
        rows = np.unique(np.concatenate([edges, g.choice(N, 192, replace=False)]))
        q, k, v = (oracle.bf16_bits_to_f64(bits[:, j, h]) for j in range(3))
        want = oracle.linear_attention(q, k, v, rows=rows)
        compare(got[rows, h], oracle.round_bf16(want), what=f"linear head {h}")
    compare(got[:, H - 1], oracle.round_bf16(np.tile(v_last.mean(0), (N, 1))), what="mean")


def test_variant_validation():
    import ctypes
    lib = vpb.lib()
    for bad in (16, 8 | 2, 8 | 4):
        dm = vpb.dims(300, variant=bad)
        size = ctypes.c_size_t(0)
        assert lib.vp_workspace_size(ctypes.byref(dm), 0, ctypes.byref(size)) == 1
