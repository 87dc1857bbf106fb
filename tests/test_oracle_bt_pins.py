"""Pins of the backbone-translator oracle (App. C.2 inside Def. 3.1). CPU only.

The oracle is checked against what the mathematics fixes: layer-norm and
attention invariants, torch's own layer-norm / attention / MLP routines on
tiny shapes, equivariance under a permutation of the source heads, invariance
to per-row shifts and scalings of the source rows, closed forms when the
residual branches are zero, and the gate's selection rules."""
import numpy as np
import pytest

import oracle
import synth

torch = pytest.importorskip("torch")
F = torch.nn.functional

pytestmark = pytest.mark.filterwarnings("ignore")

# L_s 4 -> L_t 5 (depth-ratio map 0,1,2,2,3), P = 3 source heads of 8, D_t = 2 x 8,
# E = 2, window = target layers 1..3 (source layers 1, 2, 2), d = 8, 2 heads, FFN 16.
TINY = synth.Workload("bt_tiny", 4, 3, 8, 5, 2, 8, 2, 0, 2, 6, "fp32", (6, 4),
                      bt=(1, 3, 8, 2, 16))


def _weights(wl, blob):
    """Blob tensors as float64 arrays keyed by (x, name, expert, slot)."""
    W = {}
    for (x, name, m, r, off, n, _, _) in synth.bt_blob_offsets(wl):
        W[(x, name, m, r)] = blob[off:off + n].astype(np.float64)
    return W


def _set(wl, blob, fn):
    """Copy of the blob with fn(x, name, m, r, array) -> new array applied."""
    out = blob.copy()
    for (x, name, m, r, off, n, _, _) in synth.bt_blob_offsets(wl):
        new = fn(x, name, m, r, out[off:off + n].astype(np.float64))
        if new is not None:
            out[off:off + n] = np.asarray(new, dtype=np.float64).astype(out.dtype)
    return out


def _window(wl, cache, b, s):
    """Source rows of the window for token (b, s): [N][P][d_s]."""
    lm = oracle.depth_ratio_map(wl.n_layers_src, wl.n_layers_tgt)
    return np.stack([cache[lm[t], b, :, s, :] for t in wl.bt_window]).astype(np.float64)


def _tokens(wl):
    tb = np.concatenate([np.full(L, b) for b, L in enumerate(wl.seq_lens)]).astype(np.int32)
    ts = np.concatenate([np.arange(L) for L in wl.seq_lens]).astype(np.int32)
    return tb, ts


def _inputs(wl, seed=0):
    return synth.gen_cache(wl, 0, seed), synth.gen_cache(wl, 1, seed), synth.gen_weights(wl, seed)


def _torch_backbone(wl, W, X, m, xwin, zero_branches=False):
    """The App. C.2 backbone assembled from torch's library modules (float64)."""
    P, ds, Dt = wl.src_kv_heads, wl.src_head_dim, wl.d_tgt
    _, N, d, na, df = wl.bt
    t = lambda a: torch.tensor(a, dtype=torch.float64)

    def ln(n, g, b):
        mod = torch.nn.LayerNorm(n, eps=1e-5, dtype=torch.float64)
        mod.weight.data, mod.bias.data = t(g), t(b)
        return mod

    def lin(n_in, n_out, w, b):
        mod = torch.nn.Linear(n_in, n_out, dtype=torch.float64)
        mod.weight.data, mod.bias.data = t(w).reshape(n_out, n_in), t(b)
        return mod

    g = lambda name, r=-1: W[(X, name, m, r)]
    with torch.no_grad():
        ln_in = ln(ds, g("lnin_g"), g("lnin_b"))
        lin_in = lin(ds, d, g("win"), g("bin"))
        z = F.gelu(lin_in(ln_in(t(xwin))))            # [N, P, d]
        h = z[0]
        ln_out = ln(P * d, g("lnout_g"), g("lnout_b"))
        lin_out = lin(P * d, Dt, g("wout"), g("bout"))
        Y, H = [], []
        for r in range(N):
            lnq, lnc = ln(d, g("lnq_g", r), g("lnq_b", r)), ln(d, g("lnc_g", r), g("lnc_b", r))
            mha = torch.nn.MultiheadAttention(d, na, batch_first=True, dtype=torch.float64)
            mha.in_proj_weight.data = t(np.concatenate([g("wq", r), g("wk", r), g("wv", r)])).reshape(3 * d, d)
            mha.in_proj_bias.data = t(np.concatenate([g("bq", r), g("bk", r), g("bv", r)]))
            mha.out_proj.weight.data = t(g("wo", r)).reshape(d, d)
            mha.out_proj.bias.data = t(g("bo", r))
            c = lnc(z[r])[None]
            a = mha(lnq(h)[None], c, c, need_weights=False)[0][0]
            lnf = ln(d, g("lnf_g", r), g("lnf_b", r))
            f1, f2 = lin(d, df, g("wf1", r), g("bf1", r)), lin(df, d, g("wf2", r), g("bf2", r))
            if zero_branches:
                a = torch.zeros_like(a)
            ht = h + a
            ff = f2(F.gelu(f1(lnf(ht))))
            h = ht + (torch.zeros_like(ff) if zero_branches else ff)
            H.append(h.numpy().copy())
            Y.append(F.gelu(lin_out(ln_out(h.reshape(-1)))).numpy())
    return np.stack(Y), np.stack(H)


# ---- layer norm ------------------------------------------------------------

def test_layernorm_invariants_and_library():
    rng = np.random.default_rng(0)
    x = rng.normal(size=37) * 3 + 1.5
    y = oracle.layernorm(x)
    assert abs(y.mean()) < 1e-14
    v = x.var()
    assert y.var() == pytest.approx(v / (v + 1e-5), rel=1e-12)
    # shift invariance is exact; scale invariance up to the eps term
    np.testing.assert_allclose(oracle.layernorm(x + 7.25), y, atol=1e-12)
    np.testing.assert_allclose(oracle.layernorm(4.0 * x), y, atol=1e-5)
    g, b = rng.normal(size=37), rng.normal(size=37)
    np.testing.assert_allclose(oracle.layernorm(x, g, b), g * y + b, atol=1e-13)
    np.testing.assert_array_equal(oracle.layernorm(np.full(5, 2.5), None, np.arange(5.0)),
                                  np.arange(5.0))
    ref = F.layer_norm(torch.tensor(x), (37,), torch.tensor(g), torch.tensor(b), eps=1e-5)
    np.testing.assert_allclose(oracle.layernorm(x, g, b), ref.numpy(), atol=1e-13)


# ---- attention -------------------------------------------------------------

@pytest.mark.parametrize("P,d,heads", [(3, 8, 2), (12, 32, 4), (2, 16, 1), (5, 12, 3)])
def test_attention_against_library(P, d, heads):
    rng = np.random.default_rng(P * 100 + d)
    q, k, v = (rng.normal(size=(P, d)) * 2 for _ in range(3))
    o = oracle.bt_attention(q, k, v, heads)
    dh = d // heads
    th = lambda a: torch.tensor(a).reshape(P, heads, dh).transpose(0, 1)
    ref = F.scaled_dot_product_attention(th(q), th(k), th(v)).transpose(0, 1).reshape(P, d)
    np.testing.assert_allclose(o, ref.numpy(), atol=1e-13)


def test_attention_closed_forms():
    rng = np.random.default_rng(1)
    P, d = 6, 8
    q, k, v = (rng.normal(size=(P, d)) for _ in range(3))
    # zero keys: every score equal, every query gets the mean of the values
    o = oracle.bt_attention(q, np.zeros((P, d)), v, 2)
    np.testing.assert_allclose(o, np.broadcast_to(v.mean(0), (P, d)), atol=1e-14)
    # a single key: the softmax is 1, the output is the value row
    np.testing.assert_allclose(oracle.bt_attention(q[:1], k[:1], v[:1], 4), v[:1], atol=0)
    # permuting the queries permutes the rows; permuting keys with values changes nothing
    perm = rng.permutation(P)
    base = oracle.bt_attention(q, k, v, 2)
    np.testing.assert_allclose(oracle.bt_attention(q[perm], k, v, 2), base[perm], atol=1e-14)
    np.testing.assert_allclose(oracle.bt_attention(q, k[perm], v[perm], 2), base, atol=1e-14)
    # one dominant key per head picks that value (head 0 -> key 2, head 1 -> key 4)
    k2 = np.zeros((P, d))
    k2[2, :4] = 100.0
    k2[4, 4:] = 100.0
    q2 = np.ones((P, d))
    o2 = oracle.bt_attention(q2, k2, v, 2)
    np.testing.assert_allclose(o2[:, :4], np.broadcast_to(v[2, :4], (P, 4)), atol=1e-12)
    np.testing.assert_allclose(o2[:, 4:], np.broadcast_to(v[4, 4:], (P, 4)), atol=1e-12)


# ---- one backbone ----------------------------------------------------------

@pytest.mark.parametrize("X,m", [(0, 0), (0, 1), (1, 0), (1, 1)])
def test_backbone_against_library_modules(X, m):
    wl = TINY
    k, v, blob = _inputs(wl)
    W = _weights(wl, blob)
    for (b, s) in [(0, 0), (0, 5), (1, 3)]:
        xwin = _window(wl, k if X == 0 else v, b, s)
        y, h = oracle.bt_backbone(wl, blob, X, m, xwin)
        y_ref, h_ref = _torch_backbone(wl, W, X, m, xwin)
        np.testing.assert_allclose(h, h_ref, atol=1e-12, rtol=1e-12)
        np.testing.assert_allclose(y, y_ref, atol=1e-12, rtol=1e-12)


def test_zero_residual_branches_give_equal_slots():
    """W_O, b_O, W_F2, b_F2 = 0: h_r = h_0 = z_1 for every slot, so every
    slot's output is GELU(W_out LN_out(flatten(z_1)) + b_out)."""
    wl = TINY
    k, v, blob = _inputs(wl, 2)
    blob0 = _set(wl, blob, lambda x, name, m, r, a: 0 * a if name in ("wo", "bo", "wf2", "bf2") else None)
    W = _weights(wl, blob0)
    xwin = _window(wl, v, 1, 2)
    y, h = oracle.bt_backbone(wl, blob0, 1, 1, xwin)
    for r in range(1, wl.bt[1]):
        np.testing.assert_array_equal(y[r], y[0])
        np.testing.assert_array_equal(h[r], h[0])
    y_ref, _ = _torch_backbone(wl, W, 1, 1, xwin, zero_branches=True)
    np.testing.assert_allclose(y, y_ref, atol=1e-12)
    # and the state is z of the FIRST slot: changing the other slots' sources changes nothing
    xw2 = xwin.copy()
    xw2[1:] = np.random.default_rng(5).normal(size=xw2[1:].shape)
    y2, _ = oracle.bt_backbone(wl, blob0, 1, 1, xw2)
    np.testing.assert_array_equal(y2, y)


def test_source_row_shift_and_scale_invariance():
    """LN_in normalises each source-head row of d_s values: an affine change
    a * x + c (a > 0) of any row leaves the output unchanged up to the eps term."""
    wl = TINY
    k, v, blob = _inputs(wl, 3)
    xwin = _window(wl, k, 0, 4)
    y, _ = oracle.bt_backbone(wl, blob, 0, 0, xwin)
    rng = np.random.default_rng(7)
    a = rng.choice([0.5, 2.0, 4.0], size=xwin.shape[:2])[..., None]
    c = rng.normal(size=xwin.shape[:2])[..., None] * 3
    y2, _ = oracle.bt_backbone(wl, blob, 0, 0, a * xwin + c)
    np.testing.assert_allclose(y2, y, atol=2e-4)
    # a change that is not per-row affine does change it
    x3 = xwin.copy()
    x3[0, 0, 0] += 1.0
    y3, _ = oracle.bt_backbone(wl, blob, 0, 0, x3)
    assert np.abs(y3 - y).max() > 1e-3


def test_source_head_permutation_equivariance():
    """Permuting the P source heads permutes the attention rows; with LN_out
    and W_out permuted block-wise to match (and the gate's columns), the
    translation is unchanged."""
    wl = TINY
    k, v, blob = _inputs(wl, 4)
    P, ds, Ds = wl.src_kv_heads, wl.src_head_dim, wl.d_src
    N, d = wl.bt[1], wl.bt[2]
    perm = np.array([2, 0, 1])
    kp, vp = k[:, :, perm], v[:, :, perm]
    col_pd = (perm[:, None] * d + np.arange(d)).ravel()        # flatten(h) columns
    col_win = np.concatenate([r * Ds + (perm[:, None] * ds + np.arange(ds)).ravel()
                              for r in range(N)])              # window columns

    def fn(x, name, m, r, a):
        if name in ("lnout_g", "lnout_b"):
            return a[col_pd]
        if name == "wout":
            return a.reshape(wl.d_tgt, P * d)[:, col_pd].ravel()
        if name == "wg":
            return a.reshape(wl.n_translators, N * Ds)[:, col_win].ravel()
        return None

    blob_p = _set(wl, blob, fn)
    tb, ts = _tokens(wl)
    out = oracle.bt_tokens(wl, k, v, blob, tb, ts)
    out_p = oracle.bt_tokens(wl, kp, vp, blob_p, tb, ts)
    np.testing.assert_allclose(out_p, out, atol=1e-12)
    # without the matching output permutation the result differs
    out_bad = oracle.bt_tokens(wl, kp, vp, blob, tb, ts)
    assert np.abs(out_bad - out).max() > 1e-3


# ---- the mixture -----------------------------------------------------------

def test_one_hot_gate_selects_one_backbone():
    """Wg = 0, bg = 1e4 e_m0: exp(-1e4) underflows, the softmax is one-hot and
    the output is backbone m0 alone (the construction in the proof of Prop. 3.1)."""
    wl = TINY
    k, v, blob = _inputs(wl, 5)
    tb, ts = _tokens(wl)
    for m0 in range(wl.n_translators):
        bl = _set(wl, blob, lambda x, name, m, r, a: 0 * a if name == "wg" else
                  (np.where(np.arange(a.size) == m0, 1e4, 0.0) if name == "bg" else None))
        out, g = oracle.bt_tokens(wl, k, v, bl, tb, ts, want_gate=True)
        assert (g[..., m0] == 1.0).all()
        for t in (0, 5, 7):
            for X, c in ((0, k), (1, v)):
                y, _ = oracle.bt_backbone(wl, bl, X, m0, _window(wl, c, tb[t], ts[t]))
                np.testing.assert_allclose(out[:, X, t], y, atol=1e-12)


def test_gate_reads_the_window_slot_major_head_major():
    """A gate row with one unit weight at window column c reads source value
    X_r[p][i] with c = r*D_s + p*d_s + i: g_0 = sigmoid(that value) for E = 2."""
    wl = TINY
    k, v, blob = _inputs(wl, 6)
    Ds, ds = wl.d_src, wl.src_head_dim
    tb, ts = _tokens(wl)
    for (r, p, i) in [(0, 0, 0), (2, 1, 5), (1, 2, 7)]:
        col = r * Ds + p * ds + i
        bl = _set(wl, blob, lambda x, name, m, rr, a: (np.where(np.arange(a.size) == col, 1.0, 0.0)
                                                        if name == "wg" else
                                                        (0 * a if name == "bg" else None)))
        _, g = oracle.bt_tokens(wl, k, v, bl, tb, ts, want_gate=True)
        for t in range(len(tb)):
            val = _window(wl, k, tb[t], ts[t])[r, p, i]
            assert g[0, t, 0] == pytest.approx(1.0 / (1.0 + np.exp(-val)), rel=1e-12)


def test_topk_one_is_the_argmax_backbone_and_mixture_is_linear():
    wl = TINY.replace(top_k=1)
    k, v, blob = _inputs(wl, 8)
    tb, ts = _tokens(wl)
    dense = TINY
    _, g = oracle.bt_tokens(dense, k, v, blob, tb, ts, want_gate=True)
    out1, g1 = oracle.bt_tokens(wl, k, v, blob, tb, ts, want_gate=True)
    for X, c in ((0, k), (1, v)):
        for t in range(len(tb)):
            m = int(np.argmax(g[X, t]))
            assert g1[X, t, m] == 1.0 and g1[X, t].sum() == 1.0
            y, _ = oracle.bt_backbone(wl, blob, X, m, _window(wl, c, tb[t], ts[t]))
            np.testing.assert_allclose(out1[:, X, t], y, atol=1e-12)
    # linearity in the gate weights
    n, E = len(tb), wl.n_translators
    e0 = np.zeros((2, n, E)); e0[..., 0] = 1
    e1 = np.zeros((2, n, E)); e1[..., 1] = 1
    o0 = oracle.bt_tokens(dense, k, v, blob, tb, ts, gate_fixed=e0)
    o1 = oracle.bt_tokens(dense, k, v, blob, tb, ts, gate_fixed=e1)
    om = oracle.bt_tokens(dense, k, v, blob, tb, ts, gate_fixed=0.3 * e0 + 0.7 * e1)
    np.testing.assert_allclose(om, 0.3 * o0 + 0.7 * o1, atol=1e-12)


def test_blob_size_matches_the_generator_layout():
    for name in ("bt_gpt2s_opt125m", "bt_qwen05_qwen15"):
        wl = synth.WORKLOADS[name]
        assert oracle.bt_blob_elems(wl) == wl.blob_elems()
    assert oracle.bt_blob_elems(TINY) == TINY.blob_elems()


def test_invalid_arguments_are_refused():
    wl = TINY
    k, v, blob = _inputs(wl)
    with pytest.raises(ValueError):
        oracle.bt_tokens(wl.replace(bt=(3, 3, 8, 2, 16)), k, v, blob, [0], [0])   # window past L_t
    with pytest.raises(ValueError):
        oracle.bt_tokens(wl.replace(bt=(1, 3, 8, 3, 16)), k, v, blob, [0], [0])   # d % n_a != 0
    with pytest.raises(ValueError):
        oracle.bt_tokens(wl, k, v, blob, [2], [0])                                # batch entry
