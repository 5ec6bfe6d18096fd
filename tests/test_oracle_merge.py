"""Pins of the oracle's token merging (oracle.merge): the reading of the paper's "VGGT-Prime &
Token Merging" (ToMe as used by FastVGGT, otherwise undefined).  The paper prints no merged
values, so these pin the functions to hand-built cases, conservation and a reduction."""
import numpy as np

import oracle
import synth
from oracle.layer import LN_EPS


def test_destinations_worked_example():
    # 3 views of 1 special token + 8 patches, every 3rd patch of views 1 and 2 a destination
    row_of, dst_tok = oracle.destinations(27, tokens_per_view=9, patch_start=1, stride=3)
    want = list(range(9)) + [9, 10, 13, 16] + [18, 19, 22, 25]
    assert dst_tok.tolist() == want
    assert row_of[want].tolist() == list(range(len(want)))
    assert np.all(row_of[np.setdiff1d(np.arange(27), want)] == -1)


def test_match_hand_built():
    # destinations 0, 1, 2 are e0, e1, e2; sources 3..5 lean towards 2, 0 and (equally) 1 / 2
    m = np.zeros((6, 4))
    m[0, 0] = m[1, 1] = m[2, 2] = 1.0
    m[3] = [0.1, 0.2, 0.97, 0.0]
    m[4] = [0.9, 0.1, 0.1, 0.4]
    m[5] = [0.0, 0.6, 0.6, 0.5]
    row_of = np.array([0, 1, 2, -1, -1, -1])
    assign, _ = oracle.match(m, row_of, np.array([0, 1, 2]))
    assert assign.tolist() == [0, 1, 2, 2, 0, 1]  # the tie goes to the lower row


def test_merge_conserves_mass_and_averages_members():
    g = np.random.default_rng(3)
    x = g.standard_normal((40, 16))
    assign = g.integers(0, 7, 40)
    assign[:7] = np.arange(7)  # every row has a member
    merged = oracle.merge_tokens(x, assign, 7)
    counts = np.bincount(assign, minlength=7)
    np.testing.assert_allclose((counts[:, None] * merged).sum(axis=0), x.sum(axis=0), rtol=1e-12)
    for r in range(7):
        members = [i for i in range(40) if assign[i] == r]
        np.testing.assert_allclose(merged[r], sum(x[i] for i in members) / len(members), rtol=1e-12)


def test_key_metric_is_the_unit_head_mean_of_the_keys():
    g = synth.rng(4)
    w = oracle.load_layer(synth.make_layer_weights(g, bias_std=0.05))
    x = np.random.default_rng(4).standard_normal((30, 1024))
    m = oracle.key_metric(x, w)
    k = oracle.qkv_projection(x, w, materialize=None)[:, 1].mean(axis=1)  # [N, d]
    np.testing.assert_allclose(m, k / np.linalg.norm(k, axis=1, keepdims=True), rtol=1e-10, atol=1e-12)


def test_every_token_a_destination_is_the_unmerged_block():
    # stride 1: every token is its own destination, so merging must change nothing
    g = synth.rng(6)
    w = oracle.load_layer(synth.make_layer_weights(g, block=True, bias_std=0.05, norm_jitter=0.1))
    N = 3 * 14
    x = np.random.default_rng(6).standard_normal((N, 1024))
    force = synth.forced_mix(16, 0.5)
    a, _ = oracle.global_block(x, w, force_modes=force, materialize=None, eps=LN_EPS)
    b, info = oracle.global_block(x, w, force_modes=force, materialize=None, eps=LN_EPS,
                                  merge={"stride": 1, "tokens_per_view": 14, "patch_start": 5})
    assert np.array_equal(info["merge"]["assign"], np.arange(N))
    np.testing.assert_allclose(b, a, rtol=1e-10, atol=1e-10)
