"""Pins of the replay-attention oracle (App. C.4: Top-S source-guided sparse
attention, L_Full bottom layers on full causal attention). CPU only."""
import numpy as np
import pytest

import oracle
import synth

torch = pytest.importorskip("torch")
F = torch.nn.functional

WL = synth.ReplayWorkload("replay_tiny", 4, 5, 6, 2, 16, 2, 150, (150, 97), top_s=16, n_full=1)


def _bf16(x):
    """bf16 bit patterns of values exact in bf16."""
    b = np.asarray(x, dtype=np.float32).view(np.uint32)
    assert ((b & 0xFFFF) == 0).all()
    return (b >> 16).astype(np.uint16)


def _f(bits):
    return (np.asarray(bits, dtype=np.uint32) << 16).view(np.float32).astype(np.float64)


def _numpy_topS(row_bits, u, S):
    """Library selection: sort by (value descending, position ascending), keep S."""
    vals = _f(row_bits[:u + 1])
    order = np.lexsort((np.arange(u + 1), -vals))
    return np.sort(order[:S])


def test_selection_against_numpy_sort():
    g = synth.gen_guide(WL, 3)
    rng = np.random.default_rng(0)
    for b in range(2):
        for u in list(range(0, 40)) + rng.integers(40, 150, size=40).tolist():
            got = oracle.replay_select(WL, g, b, u)
            np.testing.assert_array_equal(got, _numpy_topS(g[b, u], u, WL.top_s))


def test_selection_short_rows_ties_and_causality():
    N, S = WL.max_seq, WL.top_s
    g = np.zeros((WL.max_batch, N, N), dtype=np.uint16)
    g[0] = _bf16(np.full((N, N), 2.0))            # constant rows: the S lowest positions
    above = np.ones((N, N))
    above[np.triu_indices(N, 1)] = 2.0 ** 100
    g[1] = _bf16(above)                            # huge values above the diagonal
    for u in (0, 5, S - 1):                        # u + 1 <= S: every position
        np.testing.assert_array_equal(oracle.replay_select(WL, g, 0, u), np.arange(u + 1))
    np.testing.assert_array_equal(oracle.replay_select(WL, g, 0, 120), np.arange(S))
    for u in (S, 77, N - 1):                       # positions after u are never selected
        got = oracle.replay_select(WL, g, 1, u)
        assert got.max() <= u and got.size == S
        np.testing.assert_array_equal(got, np.arange(S))
    # a tie across the cut: 5 at {50, 55}, 3 at {10, 20, 30, 40}, 1 elsewhere; S = 5, u = 60
    row = np.ones(N)
    row[[10, 20, 30, 40]] = 3.0
    row[[50, 55]] = 5.0
    g[0, 60] = _bf16(row)
    wl2 = WL.replace(top_s=5)
    np.testing.assert_array_equal(oracle.replay_select(wl2, g, 0, 60), [10, 20, 30, 50, 55])


def _torch_attn(q, k, v, mask):
    """[Hq][N][d] outputs of torch's scaled_dot_product_attention (float64), the
    key/value heads repeated for grouped queries."""
    Hq, Hkv = q.shape[0], k.shape[0]
    kk = torch.tensor(k).repeat_interleave(Hq // Hkv, dim=0)
    vv = torch.tensor(v).repeat_interleave(Hq // Hkv, dim=0)
    return F.scaled_dot_product_attention(torch.tensor(q), kk, vv,
                                          attn_mask=torch.tensor(mask)).numpy()


def _queries(b, L, rng, n=24):
    h = rng.integers(0, WL.q_heads, size=n)
    u = np.concatenate([[0, 1, L - 1], rng.integers(0, L, size=n - 3)])
    return np.full(n, b), h, u


def test_full_layers_against_causal_library_attention():
    q, k, v = synth.gen_replay_qkv(WL, 0)
    rng = np.random.default_rng(1)
    N = WL.max_seq
    causal = np.tril(np.ones((N, N), dtype=bool))
    for b in range(2):
        ref = _torch_attn(_f(q[b]), _f(k[b]), _f(v[b]), causal)
        tb, th, tu = _queries(b, WL.seq_lens[b], rng)
        got = oracle.replay_tokens(WL, 0, q, k, v, None, tb, th, tu)   # layer 0 < n_full
        np.testing.assert_allclose(got, ref[th, tu], atol=1e-12)


def test_sparse_layers_against_masked_library_attention():
    q, k, v = synth.gen_replay_qkv(WL, 2)
    g = synth.gen_guide(WL, 1)
    rng = np.random.default_rng(2)
    N = WL.max_seq
    for b in range(2):
        mask = np.zeros((N, N), dtype=bool)
        for u in range(N):
            mask[u, _numpy_topS(g[b, u], u, WL.top_s)] = True
        ref = _torch_attn(_f(q[b]), _f(k[b]), _f(v[b]), mask)
        tb, th, tu = _queries(b, WL.seq_lens[b], rng)
        got = oracle.replay_tokens(WL, 3, q, k, v, g, tb, th, tu)      # layer 3 >= n_full
        np.testing.assert_allclose(got, ref[th, tu], atol=1e-12)
        # the guided set differs from full attention once u >= S
        full = oracle.replay_tokens(WL, 0, q, k, v, None, tb, th, tu)
        late = tu >= 2 * WL.top_s
        assert np.abs(got[late] - full[late]).max() > 1e-3


def test_layer_n_full_is_the_first_sparse_layer():
    """Layers below L_Full attend to the whole causal context; layer L_Full and
    above use the guided set (the same map gives the same result)."""
    q, k, v = synth.gen_replay_qkv(WL, 5)
    g = synth.gen_guide(WL, 4)
    tb, th, tu = _queries(1, WL.seq_lens[1], np.random.default_rng(4))
    tu = np.maximum(tu, 3 * WL.top_s)
    at_nf = oracle.replay_tokens(WL, WL.n_full, q, k, v, g, tb, th, tu)
    above = oracle.replay_tokens(WL, WL.n_full + 2, q, k, v, g, tb, th, tu)
    below = oracle.replay_tokens(WL, WL.n_full - 1, q, k, v, g, tb, th, tu)
    np.testing.assert_array_equal(at_nf, above)
    assert np.abs(at_nf - below).max() > 1e-3


def test_top_s_covering_the_context_is_full_attention():
    wl = WL.replace(top_s=WL.max_seq)
    q, k, v = synth.gen_replay_qkv(wl, 4)
    g = synth.gen_guide(wl, 2)
    tb, th, tu = _queries(0, wl.seq_lens[0], np.random.default_rng(3))
    np.testing.assert_allclose(oracle.replay_tokens(wl, 3, q, k, v, g, tb, th, tu),
                               oracle.replay_tokens(wl, 0, q, k, v, None, tb, th, tu), atol=1e-13)


def test_invalid_arguments():
    q, k, v = synth.gen_replay_qkv(WL, 0)
    g = synth.gen_guide(WL, 0)
    with pytest.raises(ValueError):
        oracle.replay_tokens(WL, 3, q, k, v, None, [0], [0], [5])        # sparse layer, no map
    with pytest.raises(ValueError):
        oracle.replay_tokens(WL, 0, q, k, v, g, [0], [WL.q_heads], [5])   # head out of range
    with pytest.raises(ValueError):
        oracle.replay_tokens(WL.replace(kv_heads=4), 0, q, k, v, g, [0], [0], [5])   # 6 % 4
