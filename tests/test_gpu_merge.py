"""GPU parity of token merging around a block's attention (vp_merge_options, the library's
reading of the paper's ToMe + VGGT-Prime combination) against the float64 oracle: the
matching (every source's destination is the most similar one, up to the metric's bf16
resolution; exact wherever the best destination leads clearly) and, with the library's
matching fed to the oracle, the stack output."""
import numpy as np
import pytest
import torch

import oracle
import synth
from tests.helpers import BF16_STEP, compare

pytestmark = pytest.mark.gpu

vpb = pytest.importorskip("paper_2609_23733_gb300.binding")

P224 = synth.tokens_per_view(224)  # 261


@pytest.fixture(scope="module", autouse=True)
def _gpu():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    vpb.lib()


def _f64(t):
    return t.detach().float().cpu().numpy().astype(np.float64)


def _check_matching(got, info, what):
    """got: the library's merged row per token; info: the oracle block's merge record."""
    mg = info["merge"]
    own, scores = mg["assign"], mg["scores"]
    dst = np.zeros(len(own), bool)
    dst[mg["dst_tok"]] = True
    assert np.array_equal(got[dst], own[dst]), what  # destinations keep their own row
    src = np.nonzero(~dst)[0]
    best = scores[src].max(axis=1)
    chosen = scores[src, got[src]]
    # the library stores the head-mean key weights and the metric rows in bf16 (relative
    # 2^-9 each, a few 1e-3 of cosine at most); the oracle's metric is exact: 2e-2 of cosine
    assert np.all(chosen >= best - 2e-2), (what, float((best - chosen).max()))
    top2 = np.sort(scores[src], axis=1)[:, -2:]
    clear = top2[:, 1] - top2[:, 0] > 4e-2
    assert clear.sum() >= 100, (what, int(clear.sum()))  # random metrics: about a third lead clearly
    assert np.array_equal(got[src][clear], own[src][clear]), what


@pytest.mark.parametrize("strides,with_qk", [((4, 10), False), ((10, 4), True)])
def test_stack_with_token_merging(strides, with_qk):
    """Two blocks over 4 views at 224 px (1,044 tokens), merging ~75 % (stride 4) and ~90 %
    (stride 10) of the tokens, routed heads in every mode."""
    N, L = 4 * P224, 2
    g = synth.rng(21)
    wts = [synth.make_layer_weights(g, block=True, bias_std=0.05, norm_jitter=0.1) for _ in range(L)]
    for w in wts:
        w["ls1"] = (0.5 * w["ls1"]).astype(np.float32)
        w["ls2"] = (0.5 * w["ls2"]).astype(np.float32)
    qs = [synth.make_qk_norm_weights(g) for _ in range(L)]
    x_bits = synth.make_tokens(21, N)
    force = np.array([[2, 1, 0, 1] * 4, synth.forced_mix(16, 0.5)])
    dm = vpb.dims(N, 16)
    dws = [vpb.to_device(w) for w in wts]
    dqs = [vpb.to_device(q) for q in qs]
    assign = [torch.full((N,), -1, dtype=torch.int32, device="cuda") for _ in range(L)]
    rope = dict(tokens_per_view=P224, patch_start=5, grid_w=16, base=100.0)
    layers = []
    for l in range(L):
        qk = vpb.qk_options(dqs[l], norm_eps=1e-6, rope=True, tokens_per_view=P224, patch_start=5, grid_w=16,
                            rope_base=100.0) if with_qk else None
        layers.append(vpb.layer_weights(dws[l], qk, vpb.merge_options(strides[l], P224, 5, assign[l])))
    ws = vpb.workspace(dm, vpb.VP_WS_STACK_MERGE)
    x = vpb.bf16_from_bits(x_bits)
    modes = torch.zeros(L, 16, dtype=torch.int32, device="cuda")
    s = torch.zeros(L, 16, device="cuda")
    vpb.vp_global_stack(dm, x, layers, torch.tensor(force, dtype=torch.int32, device="cuda"), modes, s, 1e-6, ws)
    torch.cuda.synchronize()
    assert vpb.vp_read_device_error(ws) == 0
    got_assign = [a.cpu().numpy().astype(np.int64) for a in assign]
    merge = [{"stride": st, "tokens_per_view": P224, "patch_start": 5} for st in strides]
    qk = None
    if with_qk:
        qk = [{"q_norm": (q["q_norm_g"], q["q_norm_b"]), "k_norm": (q["k_norm_g"], q["k_norm_b"]), "eps": 1e-6,
               "rope": rope} for q in qs]
    want, infos = oracle.global_stack(oracle.bf16_bits_to_f64(x_bits), [oracle.load_layer(w) for w in wts],
                                      force_modes=force, qk=qk, merge=merge, assign=got_assign)
    for l in range(L):
        _check_matching(got_assign[l], infos[l], f"block {l}")
        # the first view stays whole; later views keep 5 special tokens and every stride-th patch
        assert len(infos[l]["merge"]["dst_tok"]) == P224 + 3 * (5 + -(-256 // strides[l]))
    np.testing.assert_array_equal(modes.cpu().numpy(), force)
    compare(_f64(x), want, rel=L * BF16_STEP, what="2-block stack with token merging")


def test_merge_options_are_validated():
    N = 4 * P224
    g = synth.rng(22)
    dw = vpb.to_device(synth.make_layer_weights(g, block=True))
    x = torch.zeros(N, 1024, dtype=torch.bfloat16, device="cuda")
    modes = torch.zeros(1, 16, dtype=torch.int32, device="cuda")
    s = torch.zeros(1, 16, device="cuda")
    dm = vpb.dims(N, 16)
    small = vpb.workspace(dm, vpb.VP_WS_STACK)  # no room for the merging scratch
    with pytest.raises(vpb.VPError) as e:
        vpb.vp_global_stack(dm, x, [vpb.layer_weights(dw, None, vpb.merge_options(4, P224, 5))], None, modes,
                            s, 1e-6, small)
    assert e.value.status == 6
    ws = vpb.workspace(dm, vpb.VP_WS_STACK_MERGE)
    with pytest.raises(vpb.VPError) as e:  # views of 300 tokens do not tile N
        vpb.vp_global_stack(dm, x, [vpb.layer_weights(dw, None, vpb.merge_options(4, 300, 5))], None, modes, s,
                            1e-6, ws)
    assert e.value.status == 2
    with pytest.raises(vpb.VPError) as e:
        vpb.vp_global_stack(dm, x, [vpb.layer_weights(dw, None, vpb.merge_options(0, P224, 5))], None, modes, s,
                            1e-6, ws)
    assert e.value.status == 1


def test_single_view_merges_nothing():
    """One view: every token belongs to the first view, so every token is its own destination
    (the identity matching) and the block is the unmerged block."""
    N = P224
    g = synth.rng(23)
    w = synth.make_layer_weights(g, block=True, bias_std=0.05, norm_jitter=0.1)
    x_bits = synth.make_tokens(23, N)
    force = np.array([[2, 1, 0, 1] * 4])
    dm = vpb.dims(N, 16)
    assign = torch.full((N,), -1, dtype=torch.int32, device="cuda")
    dw = vpb.to_device(w)
    layers = [vpb.layer_weights(dw, None, vpb.merge_options(4, P224, 5, assign))]
    ws = vpb.workspace(dm, vpb.VP_WS_STACK_MERGE)
    x = vpb.bf16_from_bits(x_bits)
    modes = torch.zeros(1, 16, dtype=torch.int32, device="cuda")
    s = torch.zeros(1, 16, device="cuda")
    vpb.vp_global_stack(dm, x, layers, torch.tensor(force, dtype=torch.int32, device="cuda"), modes, s, 1e-6, ws)
    torch.cuda.synchronize()
    assert vpb.vp_read_device_error(ws) == 0
    np.testing.assert_array_equal(assign.cpu().numpy(), np.arange(N))
    want, _ = oracle.global_stack(oracle.bf16_bits_to_f64(x_bits), [oracle.load_layer(w)], force_modes=force,
                                  merge=[{"stride": 4, "tokens_per_view": P224, "patch_start": 5}])
    compare(_f64(x), want, rel=BF16_STEP, what="single view with merging on")


def test_matching_ties_go_to_the_lowest_destination():
    """View 2 repeats view 0 token for token, so every destination of view 2 has a twin in
    view 0 with the same metric row: a source whose best destination is such a pair has an
    exact tie, which goes to the lower merged row (the view-0 twin).  The twins sit in
    different 256-destination chunks, which the matching hands to different CTAs, so the tie
    is settled by the (score, lowest row) atomic maximum across CTAs."""
    N = 4 * P224
    g = synth.rng(24)
    w = synth.make_layer_weights(g, block=True, bias_std=0.05, norm_jitter=0.1)
    x_bits = synth.make_tokens(24, N)
    x_bits[2 * P224:3 * P224] = x_bits[:P224]
    dm = vpb.dims(N, 16)
    assign = torch.full((N,), -1, dtype=torch.int32, device="cuda")
    dw = vpb.to_device(w)
    layers = [vpb.layer_weights(dw, None, vpb.merge_options(4, P224, 5, assign))]
    ws = vpb.workspace(dm, vpb.VP_WS_STACK_MERGE)
    x = vpb.bf16_from_bits(x_bits)
    modes = torch.zeros(1, 16, dtype=torch.int32, device="cuda")
    s = torch.zeros(1, 16, device="cuda")
    vpb.vp_global_stack(dm, x, layers, None, modes, s, 1e-6, ws)
    torch.cuda.synchronize()
    assert vpb.vp_read_device_error(ws) == 0
    got = assign.cpu().numpy().astype(np.int64)
    row_of, dst_tok = oracle.destinations(N, P224, 5, 4)
    _, infos = oracle.global_stack(oracle.bf16_bits_to_f64(x_bits), [oracle.load_layer(w)],
                                   merge=[{"stride": 4, "tokens_per_view": P224, "patch_start": 5}],
                                   assign=[got])
    scores = infos[0]["merge"]["scores"]
    # canonical row of each merged row: a view-2 destination's twin is the view-0 token at the
    # same position, whose merged row is that position
    tok = dst_tok
    canon = np.where(tok // P224 == 2, tok % P224, np.arange(len(tok)))
    src = np.nonzero(row_of < 0)[0]
    n_ties = 0
    for i in src:
        sc = scores[i]
        best = int(np.argmax(sc))
        cls = canon == canon[best]
        others = sc[~cls]
        if sc[best] - others.max() <= 4e-2:
            continue  # no clear winner: the bf16 metric decides, not the tie rule
        want = int(np.nonzero(cls)[0].min())
        assert got[i] == want, (int(i), int(got[i]), want)
        n_ties += int(cls.sum() > 1)
    assert n_ties >= 20, n_ties


@pytest.mark.parametrize("stride", [4, 10])
def test_one_destination_takes_most_sources(stride):
    """Every source of views 1-3 is view 0's token 100 plus its own noise, so all of them join
    merged row 100 (a clear winner): one merged token of 577 (stride 4) or 691 (stride 10)
    distinct members, whose entries of the member list span many of the merge-means kernel's
    32-entry chunks (partial sums in slots, finished by the last chunk), beside rows of a single
    member; the block output is checked against the oracle with the library's matching."""
    N = 4 * P224
    g = synth.rng(25)
    w = synth.make_layer_weights(g, block=True, bias_std=0.05, norm_jitter=0.1)
    x_bits = synth.make_tokens(25, N)
    row_of, _ = oracle.destinations(N, P224, 5, stride)
    src = np.nonzero(row_of < 0)[0]
    base = synth.bf16_bits_to_f32(x_bits[100])
    noise = np.random.default_rng(25).standard_normal((len(src), x_bits.shape[1])).astype(np.float32)
    x_bits[src] = synth.f32_to_bf16_bits(base[None, :] + 0.1 * noise)
    force = np.array([[2, 1, 0, 1] * 4])
    dm = vpb.dims(N, 16)
    assign = torch.full((N,), -1, dtype=torch.int32, device="cuda")
    dw = vpb.to_device(w)
    layers = [vpb.layer_weights(dw, None, vpb.merge_options(stride, P224, 5, assign))]
    ws = vpb.workspace(dm, vpb.VP_WS_STACK_MERGE)
    x = vpb.bf16_from_bits(x_bits)
    modes = torch.zeros(1, 16, dtype=torch.int32, device="cuda")
    s = torch.zeros(1, 16, device="cuda")
    vpb.vp_global_stack(dm, x, layers, torch.tensor(force, dtype=torch.int32, device="cuda"), modes, s, 1e-6, ws)
    torch.cuda.synchronize()
    assert vpb.vp_read_device_error(ws) == 0
    got = assign.cpu().numpy().astype(np.int64)
    assert np.all(got[src] == 100)
    merge = [{"stride": stride, "tokens_per_view": P224, "patch_start": 5}]
    want, infos = oracle.global_stack(oracle.bf16_bits_to_f64(x_bits), [oracle.load_layer(w)], force_modes=force,
                                      merge=merge, assign=[got])
    _check_matching(got, infos[0], "one heavy destination")
    compare(_f64(x), want, rel=BF16_STEP, what=f"block with a merged token of {len(src) + 1} members")


def test_fewer_tokens_than_a_merge_chunk():
    """Two views of 14 tokens (5 special, 9 patches), stride 2: 28 tokens, fewer than one
    32-entry chunk of the merge-means kernel; 4 sources join the 24 destinations."""
    P, N = 14, 28
    g = synth.rng(26)
    w = synth.make_layer_weights(g, block=True, bias_std=0.05, norm_jitter=0.1)
    x_bits = synth.make_tokens(26, N)
    force = np.array([[2, 1, 0, 1] * 4])
    dm = vpb.dims(N, 16)
    assign = torch.full((N,), -1, dtype=torch.int32, device="cuda")
    dw = vpb.to_device(w)
    layers = [vpb.layer_weights(dw, None, vpb.merge_options(2, P, 5, assign))]
    ws = vpb.workspace(dm, vpb.VP_WS_STACK_MERGE)
    x = vpb.bf16_from_bits(x_bits)
    modes = torch.zeros(1, 16, dtype=torch.int32, device="cuda")
    s = torch.zeros(1, 16, device="cuda")
    vpb.vp_global_stack(dm, x, layers, torch.tensor(force, dtype=torch.int32, device="cuda"), modes, s, 1e-6, ws)
    torch.cuda.synchronize()
    assert vpb.vp_read_device_error(ws) == 0
    got = assign.cpu().numpy().astype(np.int64)
    row_of, dst_tok = oracle.destinations(N, P, 5, 2)
    assert len(dst_tok) == 24 and int((row_of < 0).sum()) == 4
    assert np.array_equal(got[row_of >= 0], row_of[row_of >= 0])
    merge = [{"stride": 2, "tokens_per_view": P, "patch_start": 5}]
    want, infos = oracle.global_stack(oracle.bf16_bits_to_f64(x_bits), [oracle.load_layer(w)], force_modes=force,
                                      merge=merge, assign=[got])
    sc = infos[0]["merge"]["scores"]
    src = np.nonzero(row_of < 0)[0]
    assert np.all(sc[src, got[src]] >= sc[src].max(axis=1) - 2e-2)  # each source at a best destination
    compare(_f64(x), want, rel=BF16_STEP, what="28-token block with merging")
