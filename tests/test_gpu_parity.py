"""GPU parity: every hot-path step through the C ABI against the float64 oracle on the
same seeded bf16 inputs.  Sizes span several tiles with ragged tails; routes must match
exactly, floating-point outputs within max-abs 2e-2 / mean-abs 2e-3."""
import numpy as np
import pytest
import torch

import oracle
import synth
from tests.helpers import BF16_STEP, calibrated_layer, compare, outside_guard

pytestmark = pytest.mark.gpu

vpb = pytest.importorskip("paper_2609_23733_gb300.binding")


@pytest.fixture(scope="module", autouse=True)
def _gpu():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    vpb.lib()  # fail loudly if the library was not built


def _bf(a):
    return vpb.bf16_from_bits(synth.f32_to_bf16_bits(a))


def _f64(t):
    return t.detach().float().cpu().numpy().astype(np.float64)


# ------------------------------------------------------------------ dense projections (a1, a9)
@pytest.mark.parametrize("M,N,K,act,with_bias,with_scale,with_res", [
    (300, 768, 256, 0, True, False, False),
    (1044, 3072, 1024, 0, True, False, False),
    (129, 1024, 1024, 0, True, True, True),
    (257, 4096, 1024, 1, True, False, False),
    (200, 1024, 4096, 0, True, True, True),
    (77, 264, 72, 1, False, True, False),
    (1, 256, 64, 0, True, False, True),
])
def test_linear_matches_oracle(M, N, K, act, with_bias, with_scale, with_res):
    g = np.random.default_rng(M * 7 + N + K)
    A = oracle.round_bf16(g.standard_normal((M, K)))
    W = oracle.round_bf16(g.uniform(-1, 1, (N, K)) * np.sqrt(6.0 / (N + K)))
    b = g.standard_normal(N).astype(np.float32) * 0.1 if with_bias else None
    sc = (1 + 0.3 * g.standard_normal(N)).astype(np.float32) if with_scale else None
    R = oracle.round_bf16(g.standard_normal((M, N))) if with_res else None
    out = vpb.vp_linear(_bf(A), _bf(W), None if b is None else torch.from_numpy(b).cuda(), act,
                        None if sc is None else torch.from_numpy(sc).cuda(),
                        None if R is None else _bf(R))
    torch.cuda.synchronize()
    ref = A @ W.T + (0 if b is None else b.astype(np.float64))
    if act == 1:
        ref = oracle.gelu(ref)
    if sc is not None:
        ref = ref * sc.astype(np.float64)
    if R is not None:
        ref = ref + R
    compare(_f64(out), oracle.round_bf16(ref), rel=BF16_STEP if with_res else 0.0, what="linear")


def test_gemm_gelu_epilogue_is_exact_to_bf16():
    # out = GELU(x) through an identity weight: the epilogue's erf (A&S 7.1.26, |error| <=
    # 1.5e-7) must give the exact GELU to within one bf16 rounding step.
    K = 256
    x = oracle.round_bf16(np.linspace(-6.0, 6.0, 300 * K).reshape(300, K))
    out = vpb.vp_linear(_bf(x), _bf(np.eye(K)), None, 1)
    torch.cuda.synchronize()
    want = oracle.gelu(x)
    got = _f64(out)
    # One bf16 step relative, plus the absolute error of the erf approximation (0.5 |x| 1.5e-7).
    assert np.all(np.abs(got - want) <= 2.0 ** -8 * np.abs(want) + 5e-7)


def test_linear_residual_in_place():
    g = np.random.default_rng(5)
    A = oracle.round_bf16(g.standard_normal((260, 512)))
    W = oracle.round_bf16(g.standard_normal((512, 512)) * 0.05)
    X = oracle.round_bf16(g.standard_normal((260, 512)))
    x = _bf(X)
    vpb.vp_linear(_bf(A), _bf(W), None, 0, None, x, out=x)
    torch.cuda.synchronize()
    compare(_f64(x), oracle.round_bf16(X + A @ W.T), rel=BF16_STEP, what="in-place residual")


# ------------------------------------------------------------------ LayerNorm (a10)
@pytest.mark.parametrize("M,D", [(1, 1024), (1000, 1024), (333, 256), (64, 4096)])
def test_layer_norm_matches_oracle(M, D):
    g = np.random.default_rng(M + D)
    X = oracle.round_bf16(g.standard_normal((M, D)) * 2 + 0.5)
    gam = (1 + 0.2 * g.standard_normal(D)).astype(np.float32)
    bet = (0.1 * g.standard_normal(D)).astype(np.float32)
    out = vpb.vp_layer_norm(_bf(X), torch.from_numpy(gam).cuda(), torch.from_numpy(bet).cuda(), 1e-6)
    torch.cuda.synchronize()
    compare(_f64(out), oracle.round_bf16(oracle.layer_norm(X, gam, bet, 1e-6)), what="layernorm")


# ------------------------------------------------------------------ router (a2, a3, a4)
def _router_case(N, H, seed, betas=None, bias_std=0.1):
    g = synth.rng(seed)
    w = synth.make_layer_weights(g, D=H * 64, H=H, bias_std=bias_std)
    qkv_bits = synth.f32_to_bf16_bits(g.standard_normal((N, 3, H, 64)).astype(np.float32))
    if betas is not None:
        w["r_beta"] = np.asarray(betas, np.float32)
    return qkv_bits, w


def _run_router(qkv_bits, w, N, H, force=None, want_r=True):
    dm = vpb.dims(N, H)
    dw = vpb.to_device(w)
    rw = vpb.router_weights(dw)
    ws = vpb.workspace(dm, vpb.VP_WS_ROUTER)
    qkv = vpb.bf16_from_bits(qkv_bits.reshape(N, -1))
    s = torch.zeros(H, device="cuda")
    modes = torch.zeros(H, dtype=torch.int32, device="cuda")
    q_pool = torch.zeros(H, 64, device="cuda")
    ctx = torch.zeros(H, 64, device="cuda")
    mean_v = torch.zeros(H, 64, device="cuda")
    r = torch.zeros(H, N, device="cuda") if want_r else None
    fm = None if force is None else torch.tensor(force, dtype=torch.int32, device="cuda")
    vpb.vp_router(dm, qkv, rw, fm, s, modes, q_pool, ctx, mean_v, r, ws)
    torch.cuda.synchronize()
    assert vpb.vp_read_device_error(ws) == 0
    out = {k: v.cpu().numpy() for k, v in dict(s=s, modes=modes, q_pool=q_pool, ctx=ctx, mean_v=mean_v).items()}
    if want_r:
        out["r"] = r.cpu().numpy()
    return out


def _oracle_router(qkv_bits, w, N, H):
    lw = oracle.load_layer(w)
    qkv = oracle.bf16_bits_to_f64(qkv_bits).reshape(N, 3, H, 64)
    res = {"s": [], "q_pool": [], "ctx": [], "mean_v": [], "r": [], "modes": []}
    for h in range(H):
        _, q_pool, r, s = oracle.layer.head_router(qkv[:, 0, h], qkv[:, 1, h], lw, h)
        res["s"].append(s)
        res["q_pool"].append(q_pool)
        res["r"].append(r)
        res["ctx"].append(r @ qkv[:, 2, h])
        res["mean_v"].append(qkv[:, 2, h].mean(0))
        res["modes"].append(oracle.select_mode(s))
    return {k: np.array(v) for k, v in res.items()}


@pytest.mark.parametrize("N,H", [(1, 16), (7, 16), (129, 5), (1044, 16), (10992, 16)])
def test_router_matches_oracle(N, H):
    betas = np.geomspace(1.0, 3000.0, H)  # spread the heads over all three bands
    qkv_bits, w = _router_case(N, H, seed=N + H, betas=betas)
    got = _run_router(qkv_bits, w, N, H)
    want = _oracle_router(qkv_bits, w, N, H)
    np.testing.assert_allclose(got["q_pool"], want["q_pool"], rtol=2e-3, atol=2e-4)
    np.testing.assert_allclose(got["s"], want["s"], rtol=2e-4, atol=1e-7)
    keep = outside_guard(want["s"])
    np.testing.assert_array_equal(got["modes"][keep], want["modes"][keep])
    np.testing.assert_allclose(got["ctx"], want["ctx"], rtol=2e-3, atol=2e-4)
    np.testing.assert_allclose(got["mean_v"], want["mean_v"], rtol=1e-4, atol=1e-5)
    np.testing.assert_allclose(got["r"], want["r"], rtol=2e-3, atol=1e-7)
    np.testing.assert_allclose(got["r"].sum(1), 1.0, atol=1e-4)
    if N >= 1044:
        assert len(set(want["modes"].tolist())) == 3  # the case exercises every route


def test_router_repeated_calls_are_bit_identical():
    """Four calls on the same device buffers at 10,992 tokens (2-3 tiles per pooling CTA, and
    Q already in L2 after the first call): bit-identical outputs.  A release of the shared-
    memory Q stage that could overtake loads still in flight once made later calls differ."""
    N, H = 10992, 16
    qkv_bits, w = _router_case(N, H, seed=31, betas=np.geomspace(1.0, 3000.0, H))
    dm = vpb.dims(N, H)
    rw = vpb.router_weights(vpb.to_device(w))
    ws = vpb.workspace(dm, vpb.VP_WS_ROUTER)
    qkv = vpb.bf16_from_bits(qkv_bits.reshape(N, -1))
    runs = []
    for _ in range(4):
        out = dict(s=torch.zeros(H, device="cuda"), modes=torch.zeros(H, dtype=torch.int32, device="cuda"),
                   q_pool=torch.zeros(H, 64, device="cuda"), ctx=torch.zeros(H, 64, device="cuda"),
                   mean_v=torch.zeros(H, 64, device="cuda"), r=torch.zeros(H, N, device="cuda"))
        vpb.vp_router(dm, qkv, rw, None, out["s"], out["modes"], out["q_pool"], out["ctx"], out["mean_v"],
                      out["r"], ws)
        torch.cuda.synchronize()
        runs.append({k: v.cpu().numpy() for k, v in out.items()})
    assert vpb.vp_read_device_error(ws) == 0
    for k in runs[0]:
        for run in runs[1:]:
            np.testing.assert_array_equal(run[k], runs[0][k], err_msg=k)


def test_router_force_modes_and_identical_keys():
    N, H = 100, 4
    g = np.random.default_rng(0)
    qkv = g.standard_normal((N, 3, H, 64)).astype(np.float32)
    qkv[:, 1] = qkv[0:1, 1]  # identical keys: s = 1/N = 0.01 exactly in real arithmetic
    qkv_bits = synth.f32_to_bf16_bits(qkv)
    w = synth.make_layer_weights(synth.rng(1), D=256, H=H)
    got = _run_router(qkv_bits, w, N, H)
    np.testing.assert_allclose(got["s"], 1.0 / N, rtol=1e-5)
    # s lands on tau_low: mean when the float32 value is <= 0.01f (it is within an ulp).
    for h in range(H):
        assert got["modes"][h] == oracle.select_mode(got["s"][h])
    forced = [2, 1, 0, 2]
    got_f = _run_router(qkv_bits, w, N, H, force=forced)
    np.testing.assert_array_equal(got_f["modes"], forced)
    np.testing.assert_allclose(got_f["s"], got["s"], rtol=0, atol=0)


# ------------------------------------------------------------------ binning (a5)
def test_bin_heads_bit_exact():
    g = np.random.default_rng(11)
    for trial in range(20):
        H = int(g.integers(1, 33))
        N = int(g.integers(1, 20000))
        modes = g.integers(0, 3, H).astype(np.int32)
        ids_o, off_o, work_o = oracle.bin_heads(modes, N)
        n_tiles = -(-N // 128)
        dm = torch.tensor(modes, device="cuda")
        ids = torch.full((H,), -1, dtype=torch.int32, device="cuda")
        off = torch.zeros(4, dtype=torch.int32, device="cuda")
        work = torch.full((H * n_tiles, 2), -1, dtype=torch.int32, device="cuda")
        nw = torch.zeros(1, dtype=torch.int32, device="cuda")
        vpb.vp_bin_heads(H, N, dm, ids, off, work, nw)
        torch.cuda.synchronize()
        np.testing.assert_array_equal(ids.cpu().numpy(), ids_o)
        np.testing.assert_array_equal(off.cpu().numpy(), off_o)
        assert int(nw.item()) == len(work_o)
        np.testing.assert_array_equal(work.cpu().numpy()[:len(work_o)], work_o)


# ------------------------------------------------------------------ head modes (a6, a7, a8)
def _run_heads(qkv_bits, w, N, H, modes, ctx, mean_v, with_saliency=False):
    dm = vpb.dims(N, H)
    dw = vpb.to_device(w)
    sw = vpb.surrogate_weights(dw)
    ws = vpb.workspace(dm, vpb.VP_WS_ROUTER)
    ids_o, off_o, _ = oracle.bin_heads(modes, N)
    y = torch.full((N, H * 64), float("nan"), dtype=torch.bfloat16, device="cuda")
    s_attn = torch.full((H,), float("nan"), device="cuda") if with_saliency else None
    vpb.vp_head_attention(dm, vpb.bf16_from_bits(qkv_bits.reshape(N, -1)),
                          torch.tensor(ids_o, device="cuda"), torch.tensor(off_o, device="cuda"),
                          torch.tensor(ctx, dtype=torch.float32, device="cuda"),
                          torch.tensor(mean_v, dtype=torch.float32, device="cuda"), sw, y, ws,
                          s_attn=s_attn)
    torch.cuda.synchronize()
    assert vpb.vp_read_device_error(ws) == 0
    out = _f64(y).reshape(N, H, 64)
    return (out, s_attn.cpu().numpy().astype(np.float64)) if with_saliency else out


def _check_saliency(s_attn, qkv, modes, what):
    """MaxAttn saliency of the full heads against the oracle's definition (same bf16 Q, K;
    the kernel's fp32 scores, sums and exponentials leave ~1e-5 relative); 0 elsewhere."""
    for h in range(len(modes)):
        if modes[h] == 2:
            want = oracle.max_attention_saliency(qkv[:, 0, h], qkv[:, 1, h])
            assert abs(s_attn[h] - want) <= 1e-3 * want, (what, h, s_attn[h], want)
        else:
            assert s_attn[h] == 0.0, (what, h, s_attn[h])


@pytest.mark.parametrize("N", [1, 5, 127, 128, 129, 300, 1044, 2000])
def test_head_modes_match_oracle(N):
    H = 6
    modes = np.array([2, 1, 0, 2, 1, 0], np.int32)
    g = synth.rng(N)
    w = synth.make_layer_weights(g, D=H * 64, H=H, bias_std=0.1)
    qkv_bits = synth.f32_to_bf16_bits(g.standard_normal((N, 3, H, 64)).astype(np.float32) * 1.5)
    lw = oracle.load_layer(w)
    qkv = oracle.bf16_bits_to_f64(qkv_bits).reshape(N, 3, H, 64)
    # The oracle's own router supplies r_h for the surrogate heads (nothing from the GPU).
    ctx, mean_v, want = np.zeros((H, 64)), np.zeros((H, 64)), np.zeros((N, H, 64))
    for h in range(H):
        Q, K, V = qkv[:, 0, h], qkv[:, 1, h], qkv[:, 2, h]
        _, _, r, _ = oracle.layer.head_router(Q, K, lw, h)
        ctx[h], mean_v[h] = r @ V, V.mean(0)
        if modes[h] == 2:
            want[:, h] = oracle.full_attention(Q, K, V)
        elif modes[h] == 1:
            mg = (lw["s_g1_w"][h], lw["s_g1_b"][h], lw["s_g2_w"][h], lw["s_g2_b"][h])
            md = (lw["s_d1_w"][h], lw["s_d1_b"][h], lw["s_d2_w"][h], lw["s_d2_b"][h])
            want[:, h], _ = oracle.surrogate_attention(V, r, mg, md)
        else:
            want[:, h], _ = oracle.mean_pooling(V)
    got, s_attn = _run_heads(qkv_bits, w, N, H, modes, ctx, mean_v, with_saliency=True)
    for h in range(H):
        compare(got[:, h], oracle.round_bf16(want[:, h]), what=f"head {h} mode {modes[h]}")
    _check_saliency(s_attn, qkv, modes, f"N={N}")


@pytest.mark.parametrize("N,modes", [(9999, [1] * 16), (4000, [1, 0] * 8), (300, [0, 1, 1, 0, 1, 1, 1, 0])])
def test_surrogate_and_mean_heads_many_items(N, modes):
    """Surrogate and mean heads over many 128-token items: every CTA takes items of several
    heads in turn, so the surrogate weights of a head are loaded into a shared-memory slot
    while the previous head's tiles still run; a ragged last item.  Every row against the
    oracle (the oracle's own router supplies r_h and C_h)."""
    H = len(modes)
    modes = np.array(modes, np.int32)
    g = synth.rng(N + H)
    w = synth.make_layer_weights(g, D=H * 64, H=H, bias_std=0.1)
    qkv_bits = synth.f32_to_bf16_bits(g.standard_normal((N, 3, H, 64)).astype(np.float32) * 1.5)
    lw = oracle.load_layer(w)
    qkv = oracle.bf16_bits_to_f64(qkv_bits).reshape(N, 3, H, 64)
    ctx, mean_v = np.zeros((H, 64)), np.zeros((H, 64))
    want = np.zeros((N, H, 64))
    for h in range(H):
        Q, K, V = qkv[:, 0, h], qkv[:, 1, h], qkv[:, 2, h]
        _, _, r, _ = oracle.layer.head_router(Q, K, lw, h)
        ctx[h], mean_v[h] = r @ V, V.mean(0)
        if modes[h] == 1:
            mg = (lw["s_g1_w"][h], lw["s_g1_b"][h], lw["s_g2_w"][h], lw["s_g2_b"][h])
            md = (lw["s_d1_w"][h], lw["s_d1_b"][h], lw["s_d2_w"][h], lw["s_d2_b"][h])
            want[:, h], _ = oracle.surrogate_attention(V, r, mg, md)
        else:
            want[:, h], _ = oracle.mean_pooling(V)
    got = _run_heads(qkv_bits, w, N, H, modes, ctx, mean_v)
    for h in range(H):
        compare(got[:, h], oracle.round_bf16(want[:, h]), what=f"N={N} head {h} mode {modes[h]}")


@pytest.mark.parametrize("N", [5000, 9999])
def test_full_attention_many_items(N):
    # More (head, query pair) work items than CTAs: every CTA runs several items in turn and
    # reuses its TMEM, barriers and pipeline stages across them.
    H = 16
    g = np.random.default_rng(N)
    qkv = g.standard_normal((N, 3, H, 64)).astype(np.float32)
    qkv_bits = synth.f32_to_bf16_bits(qkv)
    w = synth.make_layer_weights(synth.rng(1), D=H * 64, H=H)
    q = oracle.bf16_bits_to_f64(qkv_bits).reshape(N, 3, H, 64)
    got = _run_heads(qkv_bits, w, N, H, np.full(H, 2, np.int32), np.zeros((H, 64)), np.zeros((H, 64)))
    rows = np.unique(np.concatenate([np.arange(0, 300), np.arange(N - 300, N),
                                     np.random.default_rng(0).choice(N, 400, replace=False)]))
    for h in range(H):
        want = oracle.full_attention(q[:, 0, h], q[:, 1, h], q[:, 2, h], rows=rows)
        compare(got[rows, h], oracle.round_bf16(want), what=f"split head {h}")


def test_full_attention_peaked_scores():
    # Large logits make the running max move late in the key sweep (lazy rescaling path).
    N, H = 1000, 2
    g = np.random.default_rng(3)
    qkv = g.standard_normal((N, 3, H, 64)).astype(np.float32)
    qkv[:, 0] *= 4.0
    qkv[:, 1] *= np.linspace(0.2, 4.0, N)[:, None, None]
    qkv_bits = synth.f32_to_bf16_bits(qkv)
    w = synth.make_layer_weights(synth.rng(0), D=H * 64, H=H)
    q = oracle.bf16_bits_to_f64(qkv_bits).reshape(N, 3, H, 64)
    got, s_attn = _run_heads(qkv_bits, w, N, H, np.array([2, 2], np.int32), np.zeros((H, 64)),
                             np.zeros((H, 64)), with_saliency=True)
    for h in range(H):
        compare(got[:, h], oracle.round_bf16(oracle.full_attention(q[:, 0, h], q[:, 1, h], q[:, 2, h])),
                what=f"peaked head {h}")
    # the row maxima move after the first key tiles here, so the saliency needs the true row
    # maximum, not the lazily updated reference of the exponentials
    _check_saliency(s_attn, q, [2, 2], "peaked")


def test_max_attention_saliency_closed_forms():
    """Identical keys: every entry of A is 1/N.  One key scored g above the others for every
    query: s = 1 / (1 + (N - 1) e^-g).  Both at sizes spanning several key tiles."""
    H, N = 2, 1000
    g = np.random.default_rng(21)
    qkv = np.zeros((N, 3, H, 64), np.float32)
    qkv[:, 0] = g.standard_normal((N, H, 64))
    qkv[:, 1, 0] = g.standard_normal(64)          # head 0: identical keys
    qkv[:, 0, 1] = 0.0
    qkv[:, 0, 1, 0] = 8.0                         # head 1: score = k_j[0]
    qkv[777, 1, 1, 0] = 2.5                       # one key 2.5 above the rest (0)
    qkv[:, 2] = g.standard_normal((N, H, 64))
    w = synth.make_layer_weights(synth.rng(0), D=H * 64, H=H)
    _, s_attn = _run_heads(synth.f32_to_bf16_bits(qkv), w, N, H, np.array([2, 2], np.int32),
                           np.zeros((H, 64)), np.zeros((H, 64)), with_saliency=True)
    assert abs(s_attn[0] - 1.0 / N) <= 1e-5 / N
    want = 1.0 / (1.0 + (N - 1) * np.exp(-2.5))
    assert abs(s_attn[1] - want) <= 1e-5 * want


# ------------------------------------------------------------------ whole layer
def _run_layer(x_bits, w, N, H, force=None):
    dm = vpb.dims(N, H)
    dw = vpb.to_device(w)
    ws = vpb.workspace(dm, vpb.VP_WS_LAYER)
    D = H * 64
    out = torch.zeros(N, D, dtype=torch.bfloat16, device="cuda")
    s = torch.zeros(H, device="cuda")
    s_attn = torch.full((H,), float("nan"), device="cuda")
    modes = torch.zeros(H, dtype=torch.int32, device="cuda")
    fm = None if force is None else torch.tensor(force, dtype=torch.int32, device="cuda")
    vpb.vp_moh_global_attention(dm, vpb.bf16_from_bits(x_bits), dw["w_qkv"], dw["b_qkv"], dw["w_o"],
                                dw["b_o"], vpb.router_weights(dw), vpb.surrogate_weights(dw), fm, out,
                                None, None, s, modes, ws, s_attn_out=s_attn)
    torch.cuda.synchronize()
    assert vpb.vp_read_device_error(ws) == 0
    _run_layer.s_attn = s_attn.cpu().numpy().astype(np.float64)
    return _f64(out), s.cpu().numpy(), modes.cpu().numpy()


@pytest.mark.parametrize("force", [None, [2] * 16, [1] * 16, [0] * 16, [2, 1, 0, 1] * 4])
def test_layer_s4_224(force):
    """Single layer, S=4 views at 224 px (1,044 tokens), Xavier weights, seed 0."""
    wl = synth.WORKLOADS["s4_layer"]
    N = wl.N
    w = synth.make_layer_weights(synth.rng(wl.seed))
    x_bits = synth.make_tokens(wl.seed, N)
    got, s, modes = _run_layer(x_bits, w, N, 16, force)
    want = oracle.moh_attention(oracle.bf16_bits_to_f64(x_bits), oracle.load_layer(w), force_modes=force)
    compare(got, want["out"], what="layer out")
    np.testing.assert_allclose(s, want["s"], rtol=2e-3)
    np.testing.assert_array_equal(modes, want["modes"])
    # MaxAttn saliency of the full heads; both sides round their own QKV to bf16, which moves
    # a score by ~1e-3 at most
    for h in range(16):
        if modes[h] == synth.MODE_FULL:
            ref = oracle.max_attention_saliency(want["qkv"][:, 0, h], want["qkv"][:, 1, h])
            assert abs(_run_layer.s_attn[h] - ref) <= 1e-2 * ref, (h, _run_layer.s_attn[h], ref)
        else:
            assert _run_layer.s_attn[h] == 0.0
    if force is None:
        # Untrained routers: every head is diffuse, saliency ~ 1/N, so every head is mean.
        assert np.all(want["natural_modes"] == synth.MODE_MEAN)


def test_layer_s8_518_calibrated():
    """Single layer, S=8 views at 518 px (10,992 tokens), routers steered so that 4 heads
    are full, 6 surrogate and 6 mean; the oracle checks sampled rows of every head."""
    wl = synth.WORKLOADS["s8_layer_biased"]
    N = wl.N
    mix = [2, 1, 1, 0, 2, 1, 0, 0, 2, 1, 1, 0, 2, 1, 0, 0]
    x_bits, w, lw = calibrated_layer(wl.seed, N, mix)
    got, s, modes = _run_layer(x_bits, w, N, 16)
    rows = np.unique(np.concatenate([np.arange(0, 130), np.arange(N - 130, N),
                                     np.random.default_rng(0).choice(N, 600, replace=False)]))
    want = oracle.moh_attention(oracle.bf16_bits_to_f64(x_bits), lw, rows=rows)
    assert list(want["modes"]) == mix
    assert np.all(outside_guard(want["s"], guard=0.05))
    np.testing.assert_array_equal(modes, want["modes"])
    np.testing.assert_allclose(s, want["s"], rtol=5e-3)
    compare(got[rows], want["out"], what="layer out (sampled rows)")


def test_full_attention_split_tail_full_size():
    """S = 100 views at 518 px (137,400 tokens), one full head among cheap ones, as in most
    layers of the stack: on 152 SMs the last round's groups are split along the keys and
    recombined.  Sampled rows from whole groups and from split groups against the oracle."""
    N, H = 137400, 16
    g = np.random.default_rng(137)
    qkv = g.standard_normal((N, 3, H, 64)).astype(np.float32)
    qkv[:, 0, 0] *= 2.0  # a sharper head
    qkv_bits = synth.f32_to_bf16_bits(qkv)
    w = synth.make_layer_weights(synth.rng(2), D=H * 64, H=H)
    modes = np.zeros(H, np.int32)
    modes[0] = 2
    q = oracle.bf16_bits_to_f64(qkv_bits[:, :, 0].reshape(N, 3, 64))
    mean_v = np.zeros((H, 64))
    got = _run_heads(qkv_bits, w, N, H, modes, np.zeros((H, 64)), mean_v)
    tail0 = 304 * 384  # first row of the last round's groups on 152 SMs (304 whole groups)
    rows = np.unique(np.concatenate([np.arange(0, 64), np.arange(tail0 - 64, tail0 + 64),
                                     np.arange(N - 64, N),
                                     np.random.default_rng(1).choice(N, 256, replace=False)]))
    want = oracle.full_attention(q[:, 0], q[:, 1], q[:, 2], rows=rows)
    compare(got[rows, 0], oracle.round_bf16(want), what="full head, N = 137,400")
