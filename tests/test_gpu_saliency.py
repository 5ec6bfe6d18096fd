"""The router-vs-exact saliency report (§3 "Head Saliency", the appendix's MaxAttn metric,
§4.1's router) on the S=8 workload's shape (10,992 tokens): the router's s_h and the
attention kernel's exact s_h^attn = max_ij A_h[i, j] for all 16 heads (every head forced
to full) against the oracle's head_router and max_attention_saliency on the same bf16 QKV,
and the report bench.py derives from the pairs (rank correlation, route table) equal to
the one derived from the oracle's pairs."""
import numpy as np
import pytest
import torch

import bench
import oracle
import synth

pytestmark = pytest.mark.gpu

vpb = pytest.importorskip("paper_2609_23733_gb300.binding")


@pytest.fixture(scope="module", autouse=True)
def _gpu():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    vpb.lib()


def test_router_and_exact_saliency_pairs_match_the_oracle():
    wl = synth.WORKLOADS["s8_layer_biased"]
    N, H = wl.N, 16
    w = synth.make_layer_weights(synth.rng(wl.seed + 500))
    w["r_beta"] = np.geomspace(1.0, 3000.0, H).astype(np.float32)  # as bench.py's report
    lw = oracle.load_layer(w)
    qkv = oracle.qkv_projection(oracle.bf16_bits_to_f64(synth.make_tokens(wl.seed, N)), lw)
    want_s = np.array([oracle.layer.head_router(qkv[:, 0, h], qkv[:, 1, h], lw, h)[3] for h in range(H)])
    want_attn = np.array([oracle.max_attention_saliency(qkv[:, 0, h], qkv[:, 1, h]) for h in range(H)])
    # the GPU on the oracle's QKV bytes: the router, then every head in full mode
    dm = vpb.dims(N, H)
    dw = vpb.to_device(w)
    ws = vpb.workspace(dm, vpb.VP_WS_ROUTER)
    qkv_dev = vpb.bf16_from_bits(synth.f32_to_bf16_bits(qkv.reshape(N, -1).astype(np.float32)))
    s = torch.zeros(H, device="cuda")
    modes = torch.zeros(H, dtype=torch.int32, device="cuda")
    vpb.vp_router(dm, qkv_dev, vpb.router_weights(dw), None, s, modes, None, None, None, None, ws)
    s_attn = torch.full((H,), float("nan"), device="cuda")
    y = torch.empty(N, H * 64, dtype=torch.bfloat16, device="cuda")
    vpb.vp_head_attention(dm, qkv_dev, torch.arange(H, dtype=torch.int32, device="cuda"),
                          torch.tensor([0, 0, 0, H], dtype=torch.int32, device="cuda"),
                          torch.zeros(H, 64, device="cuda"), torch.zeros(H, 64, device="cuda"),
                          vpb.surrogate_weights(dw), y, ws, s_attn=s_attn)
    torch.cuda.synchronize()
    assert vpb.vp_read_device_error(ws) == 0
    got_s, got_attn = s.cpu().numpy().astype(np.float64), s_attn.cpu().numpy().astype(np.float64)
    np.testing.assert_allclose(got_s, want_s, rtol=2e-4, atol=1e-9)
    np.testing.assert_allclose(got_attn, want_attn, rtol=1e-3)
    got, want = bench.saliency_agreement(got_s, got_attn), bench.saliency_agreement(want_s, want_attn)
    assert len(set(want["routes_router"])) == 3  # the router's saliencies cover all three bands
    assert got["routes_router"] == want["routes_router"]
    assert got["routes_exact"] == want["routes_exact"]
    assert got["route_table"] == want["route_table"]
    # adjacent exact saliencies closer than the kernel's 1e-3 may swap ranks: one swap moves
    # Spearman's rho by 12 / (16 (16^2 - 1)) = 0.003
    assert abs(got["spearman"] - want["spearman"]) <= 0.01
