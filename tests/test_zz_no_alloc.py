"""vp_router_noalloc: the router for callers that cannot allocate device memory (for example
a plug-in whose host framework owns the GPU's memory pool and forbids raw cudaMalloc, or a
service that must not allocate once running).  Its scratch lives in a fixed buffer inside
the library; its results must match vp_router, which uses a caller workspace.

This file is collected last on purpose, so that a run that stops at the first failure has
run every other test before it; it must also pass on its own in a fresh process."""
import numpy as np
import pytest
import torch

import synth

pytestmark = pytest.mark.gpu

vpb = pytest.importorskip("paper_2609_23733_gb300.binding")


@pytest.fixture(scope="module", autouse=True)
def _gpu():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    vpb.lib()


def _inputs(seed, N, H):
    g = synth.rng(seed)
    w = synth.make_layer_weights(g, D=H * 64, H=H, bias_std=0.1)
    w["r_beta"] = np.geomspace(1.0, 3000.0, H).astype(np.float32)  # all three routes occur
    qkv = vpb.bf16_from_bits(synth.f32_to_bf16_bits(g.standard_normal((N, 3 * H * 64)).astype(np.float32)))
    return qkv, vpb.to_device(w)


def _outputs(N, H):
    z = lambda *shape: torch.full(shape, float("nan"), device="cuda")
    return {"s": z(H), "modes": torch.full((H,), -1, dtype=torch.int32, device="cuda"),
            "q_pool": z(H, 64), "ctx": z(H, 64), "mean_v": z(H, 64), "r": z(H, N)}


def _call(fn, dm, qkv, rw, out, *ws):
    fn(dm, qkv, rw, None, out["s"], out["modes"], out["q_pool"], out["ctx"], out["mean_v"], out["r"], *ws)
    torch.cuda.synchronize()
    return {k: v.cpu().numpy() for k, v in out.items()}


def test_noalloc_router_matches_workspace_router_on_two_calls():
    H = 16
    for call, (seed, N) in enumerate([(21, 3001), (22, 10992)]):
        qkv, dw = _inputs(seed, N, H)
        rw = vpb.router_weights(dw)
        dm = vpb.dims(N, H)
        ws = vpb.workspace(dm, vpb.VP_WS_ROUTER)
        want = _call(vpb.vp_router, dm, qkv, rw, _outputs(N, H), ws)
        got = _call(vpb.vp_router_noalloc, dm, qkv, rw, _outputs(N, H))
        np.testing.assert_array_equal(got["modes"], want["modes"], err_msg=f"call {call}")
        np.testing.assert_allclose(got["s"], want["s"], rtol=2e-4, atol=1e-7, err_msg=f"call {call}")
        for k in ("q_pool", "ctx", "mean_v"):
            np.testing.assert_allclose(got[k], want[k], rtol=2e-3, atol=2e-4, err_msg=f"{k}, call {call}")
        np.testing.assert_allclose(got["r"], want["r"], rtol=2e-3, atol=1e-7, err_msg=f"call {call}")
        assert len(set(want["modes"].tolist())) == 3


def test_noalloc_router_rejects_more_heads_than_its_buffer_holds():
    N, H = 128, 33
    qkv, dw = _inputs(0, N, 16)
    with pytest.raises(vpb.VPError) as e:
        vpb.vp_router_noalloc(vpb.dims(N, H), qkv, vpb.router_weights(dw), None,
                              torch.zeros(H, device="cuda"), torch.zeros(H, dtype=torch.int32, device="cuda"),
                              None, None, None, None)
    assert e.value.status == 8  # VP_ERR_STATIC_SCRATCH
