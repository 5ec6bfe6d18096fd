"""GPU parity of the QKV step with positional information (vp_qk_options: qk-norm and 2-D
RoPE, the library's reading of Algorithm 1's undefined P) against the float64 oracle:
the QKV intermediate, one routed layer, and a two-block stack."""
import numpy as np
import pytest
import torch

import oracle
import synth
from tests.helpers import BF16_STEP, compare

pytestmark = pytest.mark.gpu

vpb = pytest.importorskip("paper_2609_23733_gb300.binding")

P224 = synth.tokens_per_view(224)  # 261 = 5 special tokens + 16 x 16 patches
ROPE = dict(tokens_per_view=P224, patch_start=5, grid_w=16, base=100.0)


@pytest.fixture(scope="module", autouse=True)
def _gpu():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    vpb.lib()


def _f64(t):
    return t.detach().float().cpu().numpy().astype(np.float64)


def _opts(dq, norm, rope):
    return vpb.qk_options(dq if norm else None, norm_eps=1e-6, rope=rope, tokens_per_view=ROPE["tokens_per_view"],
                          patch_start=ROPE["patch_start"], grid_w=ROPE["grid_w"], rope_base=ROPE["base"])


def _oracle_qk(q, norm, rope):
    return {"q_norm": (q["q_norm_g"], q["q_norm_b"]) if norm else None,
            "k_norm": (q["k_norm_g"], q["k_norm_b"]) if norm else None,
            "eps": 1e-6, "rope": ROPE if rope else None}


@pytest.mark.parametrize("norm,rope,force", [(True, True, [2, 1, 0, 1] * 4), (True, False, [2] * 16),
                                             (False, True, [2] * 16), (True, True, None)])
def test_layer_with_qk_norm_and_rope(norm, rope, force):
    """One routed layer over S = 4 views at 224 px (1,044 tokens: 8 full tiles of 128 rows
    and a ragged 20), biases on, against oracle.moh_attention with the same reading of P."""
    N, H, D = 4 * P224, 16, 1024
    g = synth.rng(11)
    w = synth.make_layer_weights(g, bias_std=0.05)
    q = synth.make_qk_norm_weights(g)
    x_bits = synth.make_tokens(11, N)
    dm = vpb.dims(N, H)
    dw = vpb.to_device(w)
    dq = vpb.to_device(q)
    ws = vpb.workspace(dm, vpb.VP_WS_LAYER)
    out = torch.zeros(N, D, dtype=torch.bfloat16, device="cuda")
    qkv = torch.zeros(N, 3 * D, dtype=torch.bfloat16, device="cuda")
    s = torch.zeros(H, device="cuda")
    modes = torch.zeros(H, dtype=torch.int32, device="cuda")
    fm = None if force is None else torch.tensor(force, dtype=torch.int32, device="cuda")
    vpb.vp_moh_global_attention(dm, vpb.bf16_from_bits(x_bits), dw["w_qkv"], dw["b_qkv"], dw["w_o"], dw["b_o"],
                                vpb.router_weights(dw), vpb.surrogate_weights(dw), fm, out, qkv, None, s,
                                modes, ws, qk=_opts(dq, norm, rope))
    torch.cuda.synchronize()
    assert vpb.vp_read_device_error(ws) == 0
    want = oracle.moh_attention(oracle.bf16_bits_to_f64(x_bits), oracle.load_layer(w), force_modes=force,
                                qk=_oracle_qk(q, norm, rope))
    # QKV: both sides round the same float64 / float32 value to bf16, one step apart at most
    compare(_f64(qkv), want["qkv"].reshape(N, 3 * D), rel=BF16_STEP, what="qkv")
    compare(_f64(out), want["out"], what="layer out")
    np.testing.assert_allclose(s.cpu().numpy(), want["s"], rtol=2e-3)
    np.testing.assert_array_equal(modes.cpu().numpy(), want["modes"])


def test_stack_with_qk_norm_and_rope():
    """Two global blocks over 2 views at 224 px with qk-norm + RoPE in every block."""
    N, L = 2 * P224, 2
    g = synth.rng(12)
    wts = [synth.make_layer_weights(g, block=True, bias_std=0.05, norm_jitter=0.1) for _ in range(L)]
    for w in wts:
        w["ls1"] = (0.5 * w["ls1"]).astype(np.float32)
        w["ls2"] = (0.5 * w["ls2"]).astype(np.float32)
    qs = [synth.make_qk_norm_weights(g) for _ in range(L)]
    x_bits = synth.make_tokens(12, N)
    force = np.array([synth.forced_mix(16, f) for f in (0.5, 1.0)])
    dm = vpb.dims(N, 16)
    dws = [vpb.to_device(w) for w in wts]
    dqs = [vpb.to_device(q) for q in qs]
    layers = [vpb.layer_weights(w, _opts(dq, True, True)) for w, dq in zip(dws, dqs)]
    ws = vpb.workspace(dm, vpb.VP_WS_STACK)
    x = vpb.bf16_from_bits(x_bits)
    modes = torch.zeros(L, 16, dtype=torch.int32, device="cuda")
    s = torch.zeros(L, 16, device="cuda")
    vpb.vp_global_stack(dm, x, layers, torch.tensor(force, dtype=torch.int32, device="cuda"), modes, s, 1e-6, ws)
    torch.cuda.synchronize()
    assert vpb.vp_read_device_error(ws) == 0
    want, _ = oracle.global_stack(oracle.bf16_bits_to_f64(x_bits), [oracle.load_layer(w) for w in wts],
                                  force_modes=force, qk=[_oracle_qk(q, True, True) for q in qs])
    compare(_f64(x), want, rel=L * BF16_STEP, what="2-block stack with qk")


def test_qk_options_are_validated():
    N, H = 4 * P224, 16
    g = synth.rng(13)
    w = synth.make_layer_weights(g)
    dw = vpb.to_device(w)
    dm = vpb.dims(N + 1, H)  # not a whole number of views
    ws = vpb.workspace(dm, vpb.VP_WS_LAYER)
    x = torch.zeros(N + 1, 1024, dtype=torch.bfloat16, device="cuda")
    out = torch.zeros_like(x)
    with pytest.raises(vpb.VPError) as e:
        vpb.vp_moh_global_attention(dm, x, dw["w_qkv"], dw["b_qkv"], dw["w_o"], dw["b_o"], vpb.router_weights(dw),
                                    vpb.surrogate_weights(dw), None, out, None, None, None, None, ws,
                                    qk=_opts(None, False, True))
    assert e.value.status == 2
    half = vpb.qk_options({"q_norm_g": torch.ones(64, device="cuda")})  # scale without shift
    with pytest.raises(vpb.VPError) as e:
        vpb.vp_moh_global_attention(vpb.dims(N, H), x[:N], dw["w_qkv"], dw["b_qkv"], dw["w_o"], dw["b_o"],
                                    vpb.router_weights(dw), vpb.surrogate_weights(dw), None, out[:N], None, None,
                                    None, None, ws, qk=half)
    assert e.value.status == 1
