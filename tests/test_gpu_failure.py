"""Failure handling on the GPU without a fault: a device wait that nothing satisfies must give
up at its time limit, report VP_ERR_DEVICE_TIMEOUT through the workspace's error word, and
leave the CUDA context usable for the next call."""
import ctypes

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


def test_wait_gives_up_at_its_limit_and_the_context_stays_usable():
    N, H = 300, 4
    dm = vpb.dims(N, H)
    ws = vpb.workspace(dm, vpb.VP_WS_ROUTER)
    assert vpb.vp_read_device_error(ws) == 0
    limit_ns = 50_000_000  # 50 ms instead of the kernels' 4 s
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    a.record()
    vpb.vp_selftest_wait_timeout(ws, limit_ns)
    b.record()
    torch.cuda.synchronize()
    ms = a.elapsed_time(b)
    assert 50.0 <= ms < 2050.0, ms  # the limit, plus at most a few of the wait's time checks
    bits = ctypes.c_uint32(0)
    status = vpb.lib().vp_read_device_error(ctypes.c_void_p(ws.data_ptr()), ws.numel(), ctypes.byref(bits),
                                            None)
    assert status == 5 and bits.value == 1  # VP_ERR_DEVICE_TIMEOUT; VP_DEVERR_WAIT_TIMEOUT only
    assert vpb.vp_read_device_error(ws) == 0  # the read cleared the word
    # the same context and workspace still run the method: a router call against the oracle
    g = synth.rng(31)
    w = synth.make_layer_weights(g, D=H * 64, H=H)
    qkv_bits = synth.f32_to_bf16_bits(g.standard_normal((N, 3, H, 64)).astype(np.float32))
    dw = vpb.to_device(w)
    s = torch.zeros(H, device="cuda")
    modes = torch.zeros(H, dtype=torch.int32, device="cuda")
    vpb.vp_router(dm, vpb.bf16_from_bits(qkv_bits.reshape(N, -1)), vpb.router_weights(dw), None, s, modes,
                  None, None, None, None, ws)
    torch.cuda.synchronize()
    assert vpb.vp_read_device_error(ws) == 0
    lw = oracle.load_layer(w)
    qkv = oracle.bf16_bits_to_f64(qkv_bits).reshape(N, 3, H, 64)
    want = [oracle.head_router(qkv[:, 0, h], qkv[:, 1, h], lw, h)[3] for h in range(H)]
    np.testing.assert_allclose(s.cpu().numpy(), want, rtol=2e-4, atol=1e-7)


@pytest.mark.parametrize("where", ["key", "query"])
def test_nan_saliency_routes_to_full_and_sets_its_error_bit(where):
    """A NaN saliency matches no case of §4.2's routing equation; the library routes that head
    to full (the exact operator) and sets VP_DEVERR_NAN_SALIENCY.  A NaN in one key makes the
    head's routing-attention sum NaN; a NaN in one query makes its pooled query NaN.  The other
    heads are unaffected and keep the oracle's routes."""
    N, H, bad = 700, 8, 3
    g = synth.rng(33)
    w = synth.make_layer_weights(g, D=H * 64, H=H)
    w["r_beta"] = np.geomspace(1.0, 3000.0, H).astype(np.float32)
    qkv_bits = synth.f32_to_bf16_bits(g.standard_normal((N, 3, H, 64)).astype(np.float32))
    qkv_bits[123, 1 if where == "key" else 0, bad, 7] = 0x7FC0
    dm = vpb.dims(N, H)
    ws = vpb.workspace(dm, vpb.VP_WS_ROUTER)
    s = torch.zeros(H, device="cuda")
    modes = torch.full((H,), -1, dtype=torch.int32, device="cuda")
    vpb.vp_router(dm, vpb.bf16_from_bits(qkv_bits.reshape(N, -1)), vpb.router_weights(vpb.to_device(w)), None,
                  s, modes, None, None, None, None, ws)
    torch.cuda.synchronize()
    bits = ctypes.c_uint32(0)
    status = vpb.lib().vp_read_device_error(ctypes.c_void_p(ws.data_ptr()), ws.numel(), ctypes.byref(bits),
                                            None)
    assert status == 0 and bits.value == 2  # VP_DEVERR_NAN_SALIENCY alone: not a timeout
    s, modes = s.cpu().numpy(), modes.cpu().numpy()
    assert np.isnan(s[bad]) and modes[bad] == synth.MODE_FULL
    lw = oracle.load_layer(w)
    qkv = oracle.bf16_bits_to_f64(qkv_bits)
    for h in range(H):
        want = oracle.head_router(qkv[:, 0, h], qkv[:, 1, h], lw, h)[3]
        assert modes[h] == oracle.select_mode(want)
        if h != bad:
            assert abs(s[h] - want) <= 2e-4 * want, (h, s[h], want)
    assert vpb.vp_read_device_error(ws) == 0
