"""vp_router_noalloc: the router for callers that cannot allocate device memory (for example
a plug-in whose host framework owns the GPU's memory pool and forbids raw cudaMalloc, or a
service that must not allocate once running).  Its scratch lives in a fixed buffer inside
the library; its results must match vp_router, which uses a caller workspace, and the oracle.

This file is collected last on purpose, so that a run that stops at the first failure has
run every other test before it; it must also pass on its own in a fresh process."""
import numpy as np
import pytest
import torch

import oracle
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
    qkv_bits = synth.f32_to_bf16_bits(g.standard_normal((N, 3 * H * 64)).astype(np.float32))
    return qkv_bits, w


def _outputs(N, H):
    z = lambda *shape: torch.full(shape, float("nan"), device="cuda")
    return {"s": z(H), "modes": torch.full((H,), -1, dtype=torch.int32, device="cuda"),
            "q_pool": z(H, 64), "ctx": z(H, 64), "mean_v": z(H, 64), "r": z(H, N)}


def _call(fn, dm, qkv, rw, out, *ws):
    fn(dm, qkv, rw, None, out["s"], out["modes"], out["q_pool"], out["ctx"], out["mean_v"], out["r"], *ws)
    torch.cuda.synchronize()
    return {k: v.cpu().numpy() for k, v in out.items()}


def _same(got, want, what):
    np.testing.assert_array_equal(got["modes"], want["modes"], err_msg=what)
    np.testing.assert_allclose(got["s"], want["s"], rtol=2e-4, atol=1e-7, err_msg=what)
    for k in ("q_pool", "ctx", "mean_v"):
        np.testing.assert_allclose(got[k], want[k], rtol=2e-3, atol=2e-4, err_msg=f"{k}, {what}")
    np.testing.assert_allclose(got["r"], want["r"], rtol=2e-3, atol=1e-7, err_msg=what)


def test_noalloc_router_matches_workspace_router_and_oracle_on_two_calls():
    H = 16
    for call, (seed, N) in enumerate([(21, 3001), (22, 10992)]):
        qkv_bits, w = _inputs(seed, N, H)
        qkv = vpb.bf16_from_bits(qkv_bits)
        dw = vpb.to_device(w)
        rw = vpb.router_weights(dw)
        dm = vpb.dims(N, H)
        ws = vpb.workspace(dm, vpb.VP_WS_ROUTER)
        want = _call(vpb.vp_router, dm, qkv, rw, _outputs(N, H), ws)
        got = _call(vpb.vp_router_noalloc, dm, qkv, rw, _outputs(N, H))
        _same(got, want, f"call {call}")
        assert len(set(want["modes"].tolist())) == 3
        assert vpb.vp_router_noalloc_error() == 0
        if call == 0:  # and against the oracle on the same bf16 inputs
            lw = oracle.load_layer(w)
            q = oracle.bf16_bits_to_f64(qkv_bits).reshape(N, 3, H, 64)
            for h in range(H):
                _, q_pool, r, s = oracle.layer.head_router(q[:, 0, h], q[:, 1, h], lw, h)
                assert abs(got["s"][h] - s) <= 2e-4 * s, (h, got["s"][h], s)
                assert got["modes"][h] == oracle.select_mode(s, np.float32(0.01), np.float32(0.2))
                np.testing.assert_allclose(got["q_pool"][h], q_pool, rtol=2e-3, atol=2e-4)
                np.testing.assert_allclose(got["ctx"][h], r @ q[:, 2, h], rtol=2e-3, atol=2e-4)


def test_noalloc_router_takes_the_variant_bits_of_vp_router():
    """The §5 mean-query-pooling ablation reaches the kernels through the fixed-buffer path."""
    N, H = 2000, 16
    qkv_bits, w = _inputs(23, N, H)
    qkv = vpb.bf16_from_bits(qkv_bits)
    rw = vpb.router_weights(vpb.to_device(w))
    dm = vpb.dims(N, H, variant=1)  # VP_VARIANT_MEAN_QPOOL
    ws = vpb.workspace(dm, vpb.VP_WS_ROUTER)
    want = _call(vpb.vp_router, dm, qkv, rw, _outputs(N, H), ws)
    got = _call(vpb.vp_router_noalloc, dm, qkv, rw, _outputs(N, H))
    _same(got, want, "mean query pooling")
    q = synth.bf16_bits_to_f32(qkv_bits).astype(np.float64).reshape(N, 3, H, 64)
    np.testing.assert_allclose(got["q_pool"], q[:, 0].mean(axis=0), rtol=2e-3, atol=2e-4)


def test_noalloc_router_reports_a_nan_saliency_through_its_error_reader():
    N, H = 1000, 16
    qkv_bits, w = _inputs(24, N, H)
    qkv_bits = qkv_bits.reshape(N, 3, H, 64).copy()
    qkv_bits[17, 1, 5, 3] = 0x7FC0  # a NaN in one key of head 5
    qkv = vpb.bf16_from_bits(qkv_bits.reshape(N, -1))
    rw = vpb.router_weights(vpb.to_device(w))
    got = _call(vpb.vp_router_noalloc, vpb.dims(N, H), qkv, rw, _outputs(N, H))
    assert np.isnan(got["s"][5]) and got["modes"][5] == synth.MODE_FULL
    assert np.all(np.isfinite(np.delete(got["s"], 5)))
    assert vpb.vp_router_noalloc_error() == 2  # VP_DEVERR_NAN_SALIENCY, then cleared
    assert vpb.vp_router_noalloc_error() == 0


def test_noalloc_router_rejects_more_heads_than_vp_router_supports():
    N, H = 128, 33
    qkv_bits, w = _inputs(0, N, 16)
    with pytest.raises(vpb.VPError) as e:
        vpb.vp_router_noalloc(vpb.dims(N, H), vpb.bf16_from_bits(qkv_bits),
                              vpb.router_weights(vpb.to_device(w)), None,
                              torch.zeros(H, device="cuda"), torch.zeros(H, dtype=torch.int32, device="cuda"),
                              None, None, None, None)
    assert e.value.status == 2  # VP_ERR_UNSUPPORTED_SHAPE, as vp_router
