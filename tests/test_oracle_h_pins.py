"""Pins of the MoT-h oracle (App. C.5): the translated activation restored
through the target's key and value projections. CPU only."""
import numpy as np
import pytest

import oracle
import synth

pytestmark = pytest.mark.filterwarnings("ignore")


def _bf16(x):
    """fp64 values that are exact in bf16, as bf16 bit patterns."""
    b = np.asarray(x, dtype=np.float32).view(np.uint32)
    assert ((b & 0xFFFF) == 0).all(), "value not exact in bf16"
    return (b >> 16).astype(np.uint16)


def _act(wl, seed=3):
    return synth.gen_cache(wl, 0, seed)   # [L_s][B][1][S][d_as]


def _tokens(wl):
    tb = np.concatenate([np.full(L, b) for b, L in enumerate(wl.seq_lens)]).astype(np.int32)
    ts = np.concatenate([np.arange(L) for L in wl.seq_lens]).astype(np.int32)
    return tb, ts


SMALL_H = synth.Workload("h_small", 3, 1, 16, 2, 2, 8, 3, 32, 2, 9, "bf16", (9, 4),
                         act_tgt=16)   # d_as = d_at = D_t = 16, H = 2 D


def _identity_blob(wl, wk, wv):
    """Every translator the identity (W1 = [I; -I], W2 = [I, -I], zero biases:
    GELU(x) - GELU(-x) = x), a random gate, and the given projections."""
    D, H = wl.d_src, wl.hidden
    assert wl.act_tgt == D and H == 2 * D
    blob = synth.gen_weights(wl, 1).copy()
    I = np.eye(D)
    w1 = _bf16(np.vstack([I, -I]).ravel())
    w2 = _bf16(np.hstack([I, -I]).ravel())
    for (l, x, t, m, off, n, _) in synth.blob_offsets(wl):
        if t == synth.T_W1:
            blob[off:off + n] = w1
        elif t == synth.T_W2:
            blob[off:off + n] = w2
        elif t in (synth.T_B1, synth.T_B2):
            blob[off:off + n] = 0
        elif t == synth.T_WK:
            blob[off:off + n] = _bf16(wk.ravel())
        elif t == synth.T_WV:
            blob[off:off + n] = _bf16(wv.ravel())
    return blob


def test_identity_mixture_with_permutation_and_scaled_projections():
    wl = SMALL_H
    D = wl.d_src
    perm = np.random.default_rng(0).permutation(D)
    wk = np.eye(D)[perm]                                   # K = a[perm]
    scale = np.array([0.5, -1.0, 2.0, 0.25] * (D // 4))
    wv = np.diag(scale)                                    # V = scale * a
    blob = _identity_blob(wl, wk, wv)
    a = _act(wl)
    tb, ts = _tokens(wl)
    k, v, ah = oracle.translate_h_tokens(wl, a, blob, tb, ts, want_act=True)
    lmap = oracle.depth_ratio_map(wl.n_layers_src, wl.n_layers_tgt)
    for l in range(wl.n_layers_tgt):
        src = np.stack([[oracle.bf16_to_double(x) for x in a[lmap[l], b, 0, s]]
                        for b, s in zip(tb, ts)])
        np.testing.assert_allclose(ah[l], src, rtol=0, atol=1e-12)
        np.testing.assert_allclose(k[l], src[:, perm], rtol=0, atol=1e-12)
        np.testing.assert_allclose(v[l], src * scale, rtol=0, atol=1e-12)


def test_restoration_is_linear_in_the_projections():
    wl = SMALL_H.replace(name="h_lin", hidden=24, act_tgt=16)
    blob = synth.gen_weights(wl, 2)
    blob2 = blob.copy()
    for (l, x, t, m, off, n, _) in synth.blob_offsets(wl):
        if t == synth.T_WK:   # x 2: exact in bf16 (exponent + 1)
            v = blob2[off:off + n].astype(np.uint32) << 16
            blob2[off:off + n] = ((v.view(np.float32) * 2).view(np.uint32) >> 16).astype(np.uint16)
    a = _act(wl)
    tb, ts = _tokens(wl)
    k1, v1 = oracle.translate_h_tokens(wl, a, blob, tb, ts)
    k2, v2 = oracle.translate_h_tokens(wl, a, blob2, tb, ts)
    np.testing.assert_allclose(k2, 2 * k1, rtol=1e-13, atol=1e-13)
    np.testing.assert_array_equal(v2, v1)


def test_mixture_matches_the_kv_oracle_and_projections_match_numpy():
    """The activation part is the KV translation's mixture with D_t -> d_at (the
    KV entry point, pinned on its own); K and V are W^K a_hat, W^V a_hat."""
    wl = synth.Workload("h_x", 2, 1, 16, 3, 2, 8, 3, 24, 2, 7, "bf16", (7, 3), act_tgt=32,
                        top_k=2)
    blob = synth.gen_weights(wl, 4)
    a = _act(wl, 5)
    tb, ts = _tokens(wl)
    k, v, ah = oracle.translate_h_tokens(wl, a, blob, tb, ts, want_act=True)
    # the same mixture weights as a KV blob: one head of width d_at out, K and V groups alike
    kv = wl.replace(name="kv_x", tgt_kv_heads=1, tgt_head_dim=wl.act_tgt, act_tgt=0)
    mix = kv.group_elems()
    per_layer = wl.group_elems()
    blocks = []
    for r in range(len(wl.translated_layers())):
        blk = blob[r * per_layer:r * per_layer + mix]
        blocks += [blk, blk]
    kv_blob = np.concatenate(blocks)
    ref = oracle.translate_tokens(kv, a, a, kv_blob, tb, ts)     # [L_t][2][n][d_at]
    np.testing.assert_allclose(ah, ref[:, 0], rtol=1e-13, atol=1e-13)
    Dt, Da = wl.d_tgt, wl.act_tgt
    for r, l in enumerate(wl.translated_layers()):
        base = r * per_layer + mix
        wk = np.array([oracle.bf16_to_double(x) for x in blob[base:base + Dt * Da]]).reshape(Dt, Da)
        wv = np.array([oracle.bf16_to_double(x)
                       for x in blob[base + Dt * Da:base + 2 * Dt * Da]]).reshape(Dt, Da)
        np.testing.assert_allclose(k[l], ah[l] @ wk.T, rtol=1e-12, atol=1e-12)
        np.testing.assert_allclose(v[l], ah[l] @ wv.T, rtol=1e-12, atol=1e-12)


def test_untranslated_layers_are_left_untouched():
    wl = SMALL_H.replace(name="h_map", layer_map=(2, -1))
    blob = synth.gen_weights(wl, 6)
    tb, ts = _tokens(wl)
    k, v = oracle.translate_h_tokens(wl, _act(wl), blob, tb, ts)
    assert np.isnan(k[1]).all() and np.isnan(v[1]).all()
    assert np.isfinite(k[0]).all() and np.isfinite(v[0]).all()
