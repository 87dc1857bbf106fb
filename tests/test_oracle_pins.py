"""Pins for the fp64 oracle: it is checked here against what the paper and the
mathematics fix, never against itself. No GPU is needed."""
import os

import numpy as np
import pytest

import oracle
import synth
import _helpers as H

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def tiny(**kw):
    base = dict(name="tiny", n_layers_src=2, src_kv_heads=2, src_head_dim=4,
                n_layers_tgt=2, tgt_kv_heads=4, tgt_head_dim=2, n_translators=2,
                hidden=16, max_batch=2, max_seq=6, dtype="fp32", seq_lens=(6, 4))
    base.update(kw)
    return synth.Workload(**base)


def random_groups(wl, seed=0, scale=1.0):
    rng = np.random.default_rng(seed)
    E, Ds, Dt, Hh = wl.n_translators, wl.d_src, wl.d_tgt, wl.hidden
    cache = {}

    def fn(l, x):
        if (l, x) not in cache:
            cache[(l, x)] = dict(
                Wg=rng.normal(size=(E, Ds)) * scale / np.sqrt(Ds), bg=rng.normal(size=E) * scale,
                W1=[rng.normal(size=(Hh, Ds)) / np.sqrt(Ds) for _ in range(E)],
                b1=[rng.normal(size=Hh) * 0.5 for _ in range(E)],
                W2=[rng.normal(size=(Dt, Hh)) / np.sqrt(Hh) for _ in range(E)],
                b2=[rng.normal(size=Dt) * 0.5 for _ in range(E)])
        return cache[(l, x)]
    return fn


def caches(wl, seed=0):
    return synth.gen_cache(wl, 0, seed), synth.gen_cache(wl, 1, seed)


# ---------------------------------------------------------------- channel map

def test_depth_ratio_properties():
    """App. C.3: pairs layers of equal relative depth, bottom with bottom and top
    with top, order preserved; equal depths map l -> l."""
    for L_s, L_t in [(24, 28), (28, 24), (12, 12), (2, 7), (7, 2), (5, 9), (40, 3)]:
        m = oracle.depth_ratio_map(L_s, L_t)
        assert m[0] == 0 and m[-1] == L_s - 1
        assert all(a <= b for a, b in zip(m, m[1:]))
        for l, s in enumerate(m):
            # nearest relative depth: |s/(L_s-1) - l/(L_t-1)| <= half a source step
            assert abs(s * (L_t - 1) - l * (L_s - 1)) * 2 <= (L_t - 1)
    for L in (1, 4, 12, 28):
        assert oracle.depth_ratio_map(L, L) == list(range(L))


def test_depth_ratio_hand_values():
    m = oracle.depth_ratio_map(24, 28)
    # l*23/27: 3 -> 2.556 -> 3; 4 -> 3.407 -> 3; 11 -> 9.370 -> 9; 10 -> 8.519 -> 9;
    # 17 -> 14.48 -> 14; 24 -> 20.44 -> 20; 27 -> 23.
    assert (m[3], m[4], m[10], m[11], m[17], m[24], m[27]) == (3, 3, 9, 9, 14, 20, 23)
    # exact half: 3 target layers over 2 source layers, l=1 -> 0.5 -> rounds up to 1
    assert oracle.depth_ratio_map(2, 3) == [0, 1, 1]
    assert oracle.depth_ratio_map(5, 1) == [0]


# ---------------------------------------------------------------- GELU / storage

def test_gelu_against_normal_table():
    rows = [l.split() for l in open(os.path.join(GOLDEN, "normal_cdf.txt")) if l[0] != "#"]
    for xs, phis in rows:
        x, phi = float(xs), float(phis)
        assert oracle.gelu(x) == pytest.approx(x * phi, rel=1e-14, abs=0)
        assert oracle.gelu(-x) == pytest.approx(-x * (1.0 - phi), rel=1e-12, abs=0)
    assert oracle.gelu(0.0) == 0.0
    assert oracle.gelu(40.0) == pytest.approx(40.0, rel=1e-15)
    assert abs(oracle.gelu(-40.0)) < 1e-300


def test_bf16_decoding():
    assert oracle.bf16_to_double(0x3F80) == 1.0
    assert oracle.bf16_to_double(0xC000) == -2.0
    assert oracle.bf16_to_double(0x3E80) == 0.25
    assert oracle.bf16_to_double(0x3FC0) == 1.5
    assert oracle.bf16_to_double(0x0000) == 0.0


# ---------------------------------------------------------------- gate

def test_gate_softmax_closed_form():
    g = oracle.gate_from_logits([0.0, np.log(3.0)])
    assert g == pytest.approx([0.25, 0.75], abs=1e-15)
    g = oracle.gate_from_logits([np.log(0.1), np.log(0.4), np.log(0.2), np.log(0.3)])
    assert g == pytest.approx([0.1, 0.4, 0.2, 0.3], abs=1e-15)
    # max subtraction: huge logits still normalise
    g = oracle.gate_from_logits([1000.0, 1000.0 + np.log(2.0)])
    assert g == pytest.approx([1 / 3, 2 / 3], abs=1e-12)   # 1000 + ln 2 carries ~1e-13 rounding
    # one-hot: exp(-1e4) underflows to exactly 0
    g = oracle.gate_from_logits([0.0, 1e4, 0.0])
    assert g.tolist() == [0.0, 1.0, 0.0]


def test_topk_renormalisation_closed_form():
    """Def. 3.1: keep the Top-K scores and renormalise over the kept set."""
    lg = np.log([0.1, 0.4, 0.2, 0.3])
    assert oracle.gate_from_logits(lg, top_k=2) == pytest.approx([0, 4 / 7, 0, 3 / 7], abs=1e-15)
    assert oracle.gate_from_logits(lg, top_k=1) == pytest.approx([0, 1, 0, 0], abs=0)
    assert oracle.gate_from_logits(lg, top_k=3) == pytest.approx([0, 4 / 9, 2 / 9, 3 / 9], abs=1e-15)
    # Top-K = E is the dense gate
    assert oracle.gate_from_logits(lg, top_k=4) == pytest.approx([0.1, 0.4, 0.2, 0.3], abs=1e-15)
    # ties: lower index wins
    assert oracle.gate_from_logits([0.0] * 4, top_k=2).tolist() == [0.5, 0.5, 0.0, 0.0]
    assert oracle.gate_from_logits([1.0, 0.0, 1.0, 0.0], top_k=1).tolist() == [1.0, 0, 0, 0]


# ---------------------------------------------------------------- closed-form translators

def _perm_groups(wl, scales, perms_in, perms_out, gate_w=None, gate_b=None, b_in=None, b_out=None):
    D, Hh, E = wl.d_src, wl.hidden, wl.n_translators

    def fn(l, x):
        tr = [H.signed_perm_translator(D, Hh, perms_in[m], perms_out[m], scales[m],
                                       None if b_in is None else b_in[m],
                                       None if b_out is None else b_out[m]) for m in range(E)]
        return dict(Wg=np.zeros((E, D)) if gate_w is None else gate_w,
                    bg=np.zeros(E) if gate_b is None else gate_b,
                    W1=[t[0] for t in tr], b1=[t[1] for t in tr],
                    W2=[t[2] for t in tr], b2=[t[3] for t in tr])
    return fn


@pytest.mark.parametrize("dtype", ["fp32", "bf16"])
def test_identity_translator_returns_input_cache(dtype):
    """GELU(x) - GELU(-x) = x: W1=[I;-I], W2=[I,-I] translates every token to
    itself, so dst[l] must be src[pi(l)] re-headed (head-major channel order)."""
    wl = tiny(dtype=dtype, n_layers_src=3, n_layers_tgt=4, layer_map=(0, 2, -1, 1),
              hidden=20, n_translators=2, max_seq=7, seq_lens=(7, 3))
    D = wl.d_src
    ident = [np.arange(D)] * 2
    blob = H.make_blob(wl, _perm_groups(wl, [1.0, 1.0], ident, ident))
    sk, sv = caches(wl, seed=3)
    dk, dv = oracle.translate_full(wl, sk, sv, blob, wl.seq_lens)
    for l, sl in enumerate(wl.layer_map):
        for dst, src in ((dk, sk), (dv, sv)):
            for b, L in enumerate(wl.seq_lens):
                for s in range(wl.max_seq):
                    row = H.dst_row(dst, l, b, s)
                    if sl < 0 or s >= L:
                        assert np.isnan(row).all()
                    else:
                        np.testing.assert_allclose(row, H.gather_src(wl, src, sl, b, s),
                                                   rtol=1e-13, atol=1e-13)


def test_permutation_translator_pins_operand_orientation():
    """W1=[P;-P], W2=[Q,-Q] gives y = Q P z: a transposed W1 or W2, or a swapped
    head/dim index, fails this with non-symmetric permutations."""
    wl = tiny(n_translators=1, hidden=16)
    D = wl.d_src
    rng = np.random.default_rng(5)
    p, q = rng.permutation(D), rng.permutation(D)
    assert not np.array_equal(np.argsort(p), p)
    blob = H.make_blob(wl, _perm_groups(wl, [1.0], [p], [q]))
    sk, sv = caches(wl, seed=4)
    dk, dv = oracle.translate_full(wl, sk, sv, blob, wl.seq_lens)
    for b, L in enumerate(wl.seq_lens):
        for s in range(L):
            z = H.gather_src(wl, sk, 1, b, s)
            np.testing.assert_allclose(H.dst_row(dk, 1, b, s), z[p][q], rtol=1e-13, atol=1e-13)


def test_bias_terms_and_signs():
    """b1 = [beta; -beta] and b2 = delta give y = z + beta + delta exactly."""
    wl = tiny(n_translators=1)
    D = wl.d_src
    beta = np.linspace(-1.0, 1.25, D)
    delta = np.linspace(0.5, -0.75, D)
    ident = [np.arange(D)]
    blob = H.make_blob(wl, _perm_groups(wl, [1.0], ident, ident, b_in=[beta], b_out=[delta]))
    sk, sv = caches(wl, seed=6)
    dk, dv = oracle.translate_full(wl, sk, sv, blob, wl.seq_lens)
    z = H.gather_src(wl, sv, 0, 1, 2)
    b_in = H.storage_to_f64(wl, H.to_storage(wl, beta))
    b_out = H.storage_to_f64(wl, H.to_storage(wl, delta))
    np.testing.assert_allclose(H.dst_row(dv, 0, 1, 2), z + b_in + b_out, rtol=1e-13, atol=1e-13)


def test_gate_closed_form_through_translation():
    """Experts y_m = alpha_m z and gate logits w_m z[c0] + beta_m: the output is
    z * sum_m alpha_m softmax(w z[c0] + beta)_m (checks gate row/column indexing)."""
    wl = tiny(n_translators=3, hidden=16)
    D, E = wl.d_src, 3
    alpha = [0.5, -1.25, 2.0]
    c0 = 5
    Wg = np.zeros((E, D)); Wg[:, c0] = [1.0, -0.5, 0.25]
    bg = np.array([0.25, -1.0, 0.5])
    ident = [np.arange(D)] * E
    blob = H.make_blob(wl, _perm_groups(wl, alpha, ident, ident, gate_w=Wg, gate_b=bg))
    sk, sv = caches(wl, seed=7)
    dk, _ = oracle.translate_full(wl, sk, sv, blob, wl.seq_lens)
    for b, L in enumerate(wl.seq_lens):
        for s in range(L):
            z = H.gather_src(wl, sk, 0, b, s)
            lg = Wg[:, c0] * z[c0] + bg
            w = np.exp(lg - lg.max()); w /= w.sum()
            np.testing.assert_allclose(H.dst_row(dk, 0, b, s), z * float(np.dot(alpha, w)),
                                       rtol=1e-12, atol=1e-12)


def test_one_hot_gate_reproduces_single_translator():
    """Proof of Prop. 3.1: with g = e_{m0} the mixture equals translator m0, and
    equals a single-translator (E = 1) run with m0's weights."""
    wl = tiny(n_translators=3)
    rnd = random_groups(wl, seed=11)
    m0 = 1

    def onehot(l, x):
        g = dict(rnd(l, x))
        g["Wg"] = np.zeros_like(g["Wg"])
        g["bg"] = np.array([0.0, 1e4, 0.0])
        return g
    blob3 = H.make_blob(wl, onehot)
    wl1 = wl.replace(n_translators=1)

    def single(l, x):
        g = rnd(l, x)
        return dict(Wg=np.zeros((1, wl.d_src)), bg=np.zeros(1), W1=[g["W1"][m0]], b1=[g["b1"][m0]],
                    W2=[g["W2"][m0]], b2=[g["b2"][m0]])
    blob1 = H.make_blob(wl1, single)
    sk, sv = caches(wl, seed=12)
    a = oracle.translate_full(wl, sk, sv, blob3, wl.seq_lens)
    b = oracle.translate_full(wl1, sk, sv, blob1, wl.seq_lens)
    for x in (0, 1):
        np.testing.assert_array_equal(a[x], b[x])


def test_single_translator_matches_library_mlp():
    """E = 1 (the single-backbone special case) is a plain two-layer MLP:
    compare with torch.nn.functional in float64."""
    torch = pytest.importorskip("torch")
    F = torch.nn.functional
    wl = tiny(n_translators=1, hidden=12, tgt_kv_heads=3, tgt_head_dim=3)
    blob = synth.gen_weights(wl, seed=2)
    grp = H.split_blob(wl, blob)
    sk, sv = caches(wl, seed=2)
    dk, dv = oracle.translate_full(wl, sk, sv, blob, wl.seq_lens)
    for l in range(wl.n_layers_tgt):
        for x, (src, dst) in enumerate(((sk, dk), (sv, dv))):
            g = grp[(l, x)]
            for b, L in enumerate(wl.seq_lens):
                z = torch.tensor(np.stack([H.gather_src(wl, src, l, b, s) for s in range(L)]))
                y = F.linear(F.gelu(F.linear(z, torch.tensor(g["W1"][0]), torch.tensor(g["b1"][0])),
                                    approximate="none"),
                             torch.tensor(g["W2"][0]), torch.tensor(g["b2"][0])).numpy()
                got = np.stack([H.dst_row(dst, l, b, s) for s in range(L)])
                np.testing.assert_allclose(got, y, rtol=1e-12, atol=1e-12)


def test_topk_through_translation():
    """Top-K = 1 picks the argmax expert; Top-K = 2 renormalises over the two kept."""
    wl = tiny(n_translators=4, hidden=16)
    D, E = wl.d_src, 4
    alpha = [0.5, -1.5, 1.25, 2.0]
    bg = np.log([0.1, 0.4, 0.2, 0.3])
    ident = [np.arange(D)] * E
    sk, sv = caches(wl, seed=8)
    for top_k, coef in ((1, -1.5), (2, -1.5 * 4 / 7 + 2.0 * 3 / 7), (4, float(np.dot(alpha, [0.1, 0.4, 0.2, 0.3])))):
        w = wl.replace(top_k=top_k)
        blob = H.make_blob(w, _perm_groups(w, alpha, ident, ident, gate_b=bg))
        dk, _ = oracle.translate_full(w, sk, sv, blob, w.seq_lens)
        z = H.gather_src(w, sk, 1, 0, 3)
        # the gate biases are rounded to fp32 in the blob: allow for that
        np.testing.assert_allclose(H.dst_row(dk, 1, 0, 3), z * coef, rtol=2e-7, atol=2e-7)


def test_topk_equal_to_E_is_dense():
    wl = tiny(n_translators=3)
    blob = synth.gen_weights(wl, seed=5)
    sk, sv = caches(wl, seed=5)
    a = oracle.translate_full(wl, sk, sv, blob, wl.seq_lens)
    b = oracle.translate_full(wl.replace(top_k=3), sk, sv, blob, wl.seq_lens)
    np.testing.assert_array_equal(a[0], b[0])
    np.testing.assert_array_equal(a[1], b[1])


# ---------------------------------------------------------------- invariants

def test_linear_in_gate_weights():
    """Eq. mot_definition is linear in the (fixed) gate weights."""
    wl = tiny(n_translators=3)
    blob = synth.gen_weights(wl, seed=9)
    sk, sv = caches(wl, seed=9)
    tb, ts = np.array([0, 0, 1, 1]), np.array([0, 5, 1, 3])
    rng = np.random.default_rng(0)
    shape = (wl.n_layers_tgt, 2, 4, 3)
    g1, g2 = rng.random(shape), rng.random(shape)
    a = 0.3
    y1 = oracle.translate_tokens(wl, sk, sv, blob, tb, ts, gate_fixed=g1)
    y2 = oracle.translate_tokens(wl, sk, sv, blob, tb, ts, gate_fixed=g2)
    y12 = oracle.translate_tokens(wl, sk, sv, blob, tb, ts, gate_fixed=a * g1 + (1 - a) * g2)
    np.testing.assert_allclose(y12, a * y1 + (1 - a) * y2, rtol=1e-12, atol=1e-12)


def test_expert_permutation_invariance():
    wl = tiny(n_translators=4)
    rnd = random_groups(wl, seed=13)
    perm = [2, 0, 3, 1]

    def permuted(l, x):
        g = rnd(l, x)
        return dict(Wg=g["Wg"][perm], bg=g["bg"][perm], W1=[g["W1"][m] for m in perm],
                    b1=[g["b1"][m] for m in perm], W2=[g["W2"][m] for m in perm],
                    b2=[g["b2"][m] for m in perm])
    sk, sv = caches(wl, seed=13)
    a = oracle.translate_full(wl, sk, sv, H.make_blob(wl, rnd), wl.seq_lens)
    b = oracle.translate_full(wl, sk, sv, H.make_blob(wl, permuted), wl.seq_lens)
    np.testing.assert_allclose(a[0], b[0], rtol=1e-12, atol=1e-12)
    np.testing.assert_allclose(a[1], b[1], rtol=1e-12, atol=1e-12)


def test_tokens_are_independent_prefix_consistency():
    """Translation is per token: a shorter sequence gives the same values on its prefix."""
    wl = tiny(n_translators=2)
    blob = synth.gen_weights(wl, seed=4)
    sk, sv = caches(wl, seed=4)
    full = oracle.translate_full(wl, sk, sv, blob, (6, 4))
    short = oracle.translate_full(wl, sk, sv, blob, (2, 1))
    for x in (0, 1):
        np.testing.assert_array_equal(short[x][:, 0, :, :2], full[x][:, 0, :, :2])
        np.testing.assert_array_equal(short[x][:, 1, :, :1], full[x][:, 1, :, :1])
        assert np.isnan(short[x][:, 0, :, 2:]).all()


@pytest.mark.parametrize("dtype", ["fp32", "bf16"])
def test_brute_force_tiny(dtype):
    """Whole-tensor restatement with numpy primitives on a tiny ragged case, with a
    non-trivial layer map, unequal head splits and E = 3."""
    from scipy.special import erf
    wl = tiny(dtype=dtype, n_layers_src=3, n_layers_tgt=3, layer_map=(2, -1, 0), n_translators=3,
              hidden=7, src_kv_heads=3, src_head_dim=2, tgt_kv_heads=2, tgt_head_dim=5,
              max_seq=5, seq_lens=(5, 2))
    blob = synth.gen_weights(wl, seed=21)
    grp = H.split_blob(wl, blob)
    sk, sv = caches(wl, seed=21)
    dk, dv = oracle.translate_full(wl, sk, sv, blob, wl.seq_lens)
    gelu = lambda u: 0.5 * u * (1 + erf(u / np.sqrt(2)))
    for l, sl in enumerate(wl.layer_map):
        for x, (src, dst) in enumerate(((sk, dk), (sv, dv))):
            if sl < 0:
                assert np.isnan(dst[l]).all()
                continue
            g = grp[(l, x)]
            Z = H.storage_to_f64(wl, src[sl]).transpose(0, 2, 1, 3).reshape(wl.max_batch, wl.max_seq, -1)
            lg = np.einsum("bsc,mc->bsm", Z, g["Wg"]) + g["bg"]
            w = np.exp(lg - lg.max(-1, keepdims=True)); w /= w.sum(-1, keepdims=True)
            Y = sum(w[..., m:m + 1] * (np.einsum("bsj,ij->bsi",
                                                  gelu(np.einsum("bsc,jc->bsj", Z, g["W1"][m]) + g["b1"][m]),
                                                  g["W2"][m]) + g["b2"][m])
                    for m in range(3))
            Y = Y.reshape(wl.max_batch, wl.max_seq, wl.tgt_kv_heads, wl.tgt_head_dim).transpose(0, 2, 1, 3)
            for b, L in enumerate(wl.seq_lens):
                np.testing.assert_allclose(dst[l, b, :, :L], Y[b, :, :L], rtol=1e-12, atol=1e-12)
                assert np.isnan(dst[l, b, :, L:]).all()


def test_invalid_arguments_rejected():
    wl = tiny()
    blob = synth.gen_weights(wl)
    sk, sv = caches(wl)
    with pytest.raises(ValueError):
        oracle.translate_full(wl, sk, sv, blob, (7, 1))           # seq_len > S_max
    with pytest.raises(ValueError):
        oracle.translate_tokens(wl, sk, sv, blob, [2], [0])       # batch index out of range
    with pytest.raises(ValueError):
        oracle.translate_full(wl.replace(layer_map=(0, 5)), sk, sv, blob, wl.seq_lens)
    with pytest.raises(ValueError):
        oracle.depth_ratio_map(0, 3)
