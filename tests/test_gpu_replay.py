"""Replay attention (App. C.4) on the GPU through the C ABI, against the fp64
oracle: the Top-S selection bit for bit, the attention within the bf16 bar."""
import numpy as np
import pytest

import oracle
import synth

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")
if not torch.cuda.is_available():
    pytest.skip("needs a CUDA GPU", allow_module_level=True)

import _gpu as G   # noqa: E402
M = G.M

RW = synth.ReplayWorkload
SMALL = {
    # GQA 12 / 2, d = 128, S = 16 (short rows below S), ragged batch
    "r_gqa6_d128": RW("r_gqa6_d128", 6, 7, 12, 2, 128, 2, 300, (300, 131), top_s=16, n_full=2),
    # no GQA, d = 64, the paper's S = 128 with rows shorter and longer than S
    "r_mha_d64": RW("r_mha_d64", 4, 4, 4, 4, 64, 3, 400, (400, 128, 129), top_s=128, n_full=1),
    # 16 query heads per key/value head, one long row per entry
    "r_gqa16": RW("r_gqa16", 2, 2, 16, 1, 64, 1, 1000, (1000,), top_s=64, n_full=1),
    # d = 128 on the tensor-core guided kernel: S = 128, 16 heads per group, ragged rows
    "r_gqa16_d128": RW("r_gqa16_d128", 2, 4, 16, 1, 128, 3, 520, (520, 127, 129), top_s=128,
                       n_full=1),
    # d = 128, no GQA, an S that is not a multiple of 4 (partial gather4 groups)
    "r_mha_d128_s99": RW("r_mha_d128_s99", 2, 4, 3, 3, 128, 2, 333, (333, 98), top_s=99, n_full=1),
}


def _dev(a):
    return torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).cuda()


class ReplayRun:
    def __init__(self, wl, seq=None, batch=None):
        self.wl = wl
        self.h = M.mot_create_replay(M.replay_config_from(wl))
        self.seq = list(wl.seq_lens if seq is None else seq)
        self.batch = len(self.seq) if batch is None else batch
        self.lens = torch.tensor(self.seq, dtype=torch.int32, device="cuda")

    def select(self, g):
        sel = torch.full((self.wl.max_batch, self.wl.max_seq, self.wl.top_s), -7,
                         dtype=torch.int32, device="cuda")
        M.mot_replay_select(self.h, _dev(g), self.lens, self.batch, sel)
        torch.cuda.synchronize()
        return sel.cpu().numpy()

    def attend(self, layer, q, k, v, g):
        out = torch.full((self.wl.max_batch, self.wl.q_heads, self.wl.max_seq, self.wl.head_dim),
                         G.SENTINEL_BF16, dtype=torch.int16, device="cuda")
        M.mot_replay_attention(self.h, layer, _dev(q), _dev(k), _dev(v),
                               None if g is None else _dev(g), self.lens, self.batch, out)
        torch.cuda.synchronize()
        return out


BF16 = synth.WORKLOADS["gpt2s_opt125m"]   # carries the bf16 tolerance of the parity bar


def _f64(bits_t):
    return bits_t.view(torch.bfloat16).double().cpu().numpy()


@pytest.mark.parametrize("name", sorted(SMALL))
def test_selection_is_bit_exact_on_every_row(name):
    wl = SMALL[name]
    g = synth.gen_guide(wl, 3)
    run = ReplayRun(wl)
    sel = run.select(g)
    for b, L in enumerate(wl.seq_lens):
        for u in range(L):
            ref = oracle.replay_select(wl, g, b, u)
            row = sel[b, u]
            np.testing.assert_array_equal(row[:ref.size], ref, err_msg=f"b={b} u={u}")
            assert (row[ref.size:] == -1).all()
        assert (sel[b, L:] == -7).all()   # rows past the sequence are not written


@pytest.mark.parametrize("name", ["r_gqa6_d128", "r_mha_d64"])   # max_seq 300 and 400: scalar and 16-byte loads
def test_selection_ties_and_constant_rows(name):
    wl = SMALL[name].replace(top_s=8)
    N = wl.max_seq
    g = np.zeros((wl.max_batch, N, N), dtype=np.uint16)
    g[0] = 0x4000                                  # every score 2.0: the lowest positions win
    rng = np.random.default_rng(0)
    g[1] = (0x3F80 + rng.integers(0, 3, size=(N, N))).astype(np.uint16)   # three values only
    if wl.batch > 2:   # mixed signs (no exact zeros: -0 and +0 order apart in the 16-bit keys)
        x = rng.standard_normal((N, N)).astype(np.float32)
        g[2] = (x.view(np.uint32) >> 16).astype(np.uint16)
    run = ReplayRun(wl)
    sel = run.select(g)
    for b, L in enumerate(wl.seq_lens):
        for u in range(0, L, 7):
            ref = oracle.replay_select(wl, g, b, u)
            np.testing.assert_array_equal(sel[b, u, :ref.size], ref)


@pytest.mark.parametrize("span", [1, 255, 256, 257, 511, 512, 4097, 0x7EFF])
def test_selection_across_key_ranges(span):
    """Rows whose 16-bit keys span `span` values: the histogram digit's width
    follows the row's range, so spans around 2^8 and 2^9 take the one-pass and
    two-pass cases and their boundary."""
    wl = SMALL["r_mha_d64"].replace(top_s=32)
    N = wl.max_seq
    rng = np.random.default_rng(span)
    base = 0x3C00 if span < 0x4000 else 0x0080        # positive bf16 bit patterns, no NaN or Inf
    g = (base + rng.integers(0, span + 1, size=(wl.max_batch, N, N))).astype(np.uint16)
    g[:, :, 0] = base                                   # the range's ends are present
    g[:, :, 1] = base + span
    run = ReplayRun(wl)
    sel = run.select(g)
    for b, L in enumerate(wl.seq_lens):
        for u in range(0, L, 5):
            ref = oracle.replay_select(wl, g, b, u)
            np.testing.assert_array_equal(sel[b, u, :ref.size], ref, err_msg=f"b={b} u={u}")


@pytest.mark.parametrize("max_seq", [4104, 4099])   # 16-byte and scalar loads
def test_selection_rows_longer_than_the_key_cache(max_seq):
    """Rows past 4,096 positions take the streaming selection (the row read once per pass)."""
    wl = RW("r_long", 2, 2, 4, 1, 64, 1, max_seq, (max_seq,), top_s=128, n_full=1)
    g = synth.gen_guide(wl, 13)
    sel = ReplayRun(wl).select(g)
    rng = np.random.default_rng(max_seq)
    for u in np.unique(np.concatenate([[0, 127, 128, 4095, 4096, max_seq - 1],
                                       rng.integers(129, max_seq, size=40)])):
        ref = oracle.replay_select(wl, g, 0, int(u))
        np.testing.assert_array_equal(sel[0, u, :ref.size], ref, err_msg=f"u={u}")


@pytest.mark.parametrize("name", sorted(SMALL))
def test_attention_matches_oracle(name):
    wl = SMALL[name]
    q, k, v = synth.gen_replay_qkv(wl, 1)
    g = synth.gen_guide(wl, 5)
    run = ReplayRun(wl)
    rng = np.random.default_rng(7)
    for layer in (0, wl.n_full, wl.n_full + 3):
        out = run.attend(layer, q, k, v, None if layer < wl.n_full else g)
        tb, th, tu = [], [], []
        for b, L in enumerate(wl.seq_lens):
            us = np.unique(np.concatenate([[0, 1, L - 1, min(L - 1, wl.top_s), min(L - 1, wl.top_s - 1)],
                                           rng.integers(0, L, size=20)]))
            for u in us:
                for h in rng.choice(wl.q_heads, size=min(4, wl.q_heads), replace=False):
                    tb.append(b); th.append(h); tu.append(u)
        ref = oracle.replay_tokens(wl, layer, q, k, v, g, tb, th, tu)
        got = _f64(out)[tb, th, tu]
        G.assert_parity(BF16, got, ref, f"{name} layer {layer}")
        o = out.cpu().numpy()
        for b, L in enumerate(wl.seq_lens):
            assert (o[b, :, L:] == np.int16(G.SENTINEL_BF16)).all()


@pytest.mark.parametrize("group", [2, 3, 4, 5, 7, 8, 12])
def test_guided_attention_every_group_size(group):
    """The tensor-core guided kernel is instantiated per GQA group size G (the
    query heads of one key/value head): a guided layer with d = 128 and S = 128
    for each G the other tests do not reach, sampled against the oracle."""
    kv = 2 if group <= 4 else 1
    wl = RW(f"r_g{group}", 2, 3, group * kv, kv, 128, 2, 264, (264, 131), top_s=128, n_full=1)
    q, k, v = synth.gen_replay_qkv(wl, 17)
    g = synth.gen_guide(wl, 19)
    run = ReplayRun(wl)
    out = run.attend(2, q, k, v, g)
    rng = np.random.default_rng(group)
    tb, th, tu = [], [], []
    for b, L in enumerate(wl.seq_lens):
        us = np.unique(np.concatenate([[0, 127, 128, L - 1], rng.integers(0, L, size=12)]))
        for u in us:
            for h in range(wl.q_heads):
                tb.append(b); th.append(h); tu.append(u)
    ref = oracle.replay_tokens(wl, 2, q, k, v, g, tb, th, tu)
    G.assert_parity(BF16, _f64(out)[tb, th, tu], ref, f"group {group}")
    o = out.cpu().numpy()
    for b, L in enumerate(wl.seq_lens):
        assert (o[b, :, L:] == np.int16(G.SENTINEL_BF16)).all()


@pytest.mark.parametrize("gain", [0.05, 2.0])
def test_attention_scores_rising_along_the_context(gain):
    """Keys that grow along a common direction of the queries, so a query's scores
    rise with the key position by about `gain` (base 2) per key: the full-attention
    kernel's running max passes its 2^8 margin on later key tiles and rescales O
    and the row sum (gain 0.05: every tile or two by a moderate factor; gain 2:
    every tile, the earlier keys' weight vanishing), and the guided kernel sees
    rows whose selected scores span hundreds of binades. Against the oracle."""
    import _helpers as H
    wl = RW("r_rise", 2, 3, 12, 2, 128, 2, 520, (520, 300), top_s=128, n_full=1)
    q, k, v = synth.gen_replay_qkv(wl, 23)
    g = synth.gen_guide(wl, 29)
    # q . k / sqrt(d) = 128 (gain j / 16) / sqrt(128) ~ 0.7 gain j, about gain j in base 2
    qf = 0.25 * H.bf16_bits_to_f64(q) + 1.0
    j = np.arange(wl.max_seq, dtype=np.float64)[None, None, :, None]
    kf = 0.25 * H.bf16_bits_to_f64(k) + gain * j / 16.0
    q = H.f32_to_bf16_bits(qf.astype(np.float32))
    k = H.f32_to_bf16_bits(kf.astype(np.float32))
    run = ReplayRun(wl)
    rng = np.random.default_rng(31)
    for layer in (0, 2):
        out = run.attend(layer, q, k, v, None if layer < wl.n_full else g)
        tb, th, tu = [], [], []
        for b, L in enumerate(wl.seq_lens):
            us = np.unique(np.concatenate([[0, 127, 128, 255, 256, L - 1], rng.integers(0, L, size=10)]))
            for u in us:
                for h in range(wl.q_heads):
                    tb.append(b); th.append(h); tu.append(u)
        ref = oracle.replay_tokens(wl, layer, q, k, v, g, tb, th, tu)
        G.assert_parity(BF16, _f64(out)[tb, th, tu], ref, f"gain {gain} layer {layer}")


def test_full_size_layer_sampled():
    """Qwen2.5-0.5B -> 1.5B replay shapes (4 x 4096 context, 12 / 2 heads of 128,
    S = 128): one full and one guided layer, in the benchmark's launch configuration."""
    wl = synth.REPLAY_WORKLOADS["replay_qwen05_qwen15"]
    q, k, v = synth.gen_replay_qkv(wl, 2)
    g = synth.gen_guide(wl, 9)
    run = ReplayRun(wl)
    sel = run.select(g)
    rng = np.random.default_rng(11)
    # 256 selection rows per batch entry (both ends, the S boundary, a whole
    # 128-row block and random rows), each bit-exact
    for b in range(wl.batch):
        blk = 128 * int(rng.integers(1, 32))
        us = np.unique(np.concatenate([[0, 127, 128, 4095], np.arange(blk, blk + 128),
                                       rng.integers(0, 4096, size=124)]))
        for u in us:
            ref = oracle.replay_select(wl, g, b, int(u))
            np.testing.assert_array_equal(sel[b, u, :ref.size], ref)
    # 2048 queries per layer: a full layer, a guided layer and the last layer;
    # every query head of one whole 128-query tile of one batch entry included
    for layer in (1, 5, wl.n_layers_tgt - 1):
        out = run.attend(layer, q, k, v, g)
        t0 = 128 * int(rng.integers(0, 32))
        tile_h, tile_u = np.meshgrid(np.arange(wl.q_heads), np.arange(t0, t0 + 128), indexing="ij")
        n = 2048 - tile_h.size
        tb = np.concatenate([np.full(tile_h.size, 3), rng.integers(0, wl.batch, size=n)])
        th = np.concatenate([tile_h.ravel(), rng.integers(0, wl.q_heads, size=n)])
        tu = np.concatenate([tile_u.ravel(), [0, 4095], rng.integers(0, 4096, size=n - 2)])
        ref = oracle.replay_tokens(wl, layer, q, k, v, g, tb, th, tu)
        G.assert_parity(BF16, _f64(out)[tb, th, tu], ref, f"full-size layer {layer}")


def test_full_layers_use_the_tensor_core_kernel():
    """max_seq % 8 == 0: full layers run the tcgen05 attention kernel (after the V
    transpose); guided layers run the selection and the gather kernel."""
    wl = SMALL["r_mha_d64"]
    q, k, v = synth.gen_replay_qkv(wl, 0)
    g = synth.gen_guide(wl, 0)
    run = ReplayRun(wl)
    M.mot_profile_enable(run.h, True)
    run.attend(0, q, k, v, None)
    run.attend(2, q, k, v, g)
    prof = M.mot_profile_read(run.h)
    assert set(prof) == {"replay_vt", "replay_fmha_full", "replay_select", "replay_attn_sparse"}


def test_batch_prefix_and_errors():
    wl = SMALL["r_mha_d64"]
    q, k, v = synth.gen_replay_qkv(wl, 0)
    g = synth.gen_guide(wl, 0)
    run = ReplayRun(wl, batch=2)
    out = run.attend(3, q, k, v, g).cpu().numpy()
    assert (out[2] == np.int16(G.SENTINEL_BF16)).all()    # entry 2 is past `batch`
    dst = torch.empty(out.shape, dtype=torch.int16, device="cuda")
    with pytest.raises(M.MotError) as e:                   # a guided layer needs its map
        M.mot_replay_attention(run.h, 3, _dev(q), _dev(k), _dev(v), None, run.lens, 2, dst)
    assert e.value.status == M.MOT_ERR_INVALID_ARG
    with pytest.raises(M.MotError) as e:
        M.mot_create_replay(M.replay_config_from(wl.replace(head_dim=96)))
    assert e.value.status == M.MOT_ERR_UNSUPPORTED
    with pytest.raises(M.MotError) as e:
        M.mot_create_replay(M.replay_config_from(wl.replace(kv_heads=3)))
    assert e.value.status == M.MOT_ERR_INVALID_ARG


def test_guided_timeout_is_reported_and_recovers():
    """Failure detection without a fault: with the stall hook the guided kernel's
    first CTA withholds one MMA completion signal, its wait runs out after the
    short limit, the kernel unwinds and the status word reports a timeout. The
    next guided layer on the same context matches the oracle."""
    wl = SMALL["r_gqa6_d128"]
    q, k, v = synth.gen_replay_qkv(wl, 3)
    g = synth.gen_guide(wl, 6)
    run = ReplayRun(wl)
    layer = wl.n_full + 1
    M.mot_debug_set(run.h, True, 20_000_000)        # about 10 ms of SM cycles
    run.attend(layer, q, k, v, g)
    assert M.mot_get_device_status(run.h) == M.MOT_ERR_TIMEOUT
    assert M.mot_get_device_status(run.h) == M.MOT_OK   # reading cleared it
    M.mot_debug_set(run.h, False, 0)
    out = run.attend(layer, q, k, v, g)
    assert M.mot_get_device_status(run.h) == M.MOT_OK
    rng = np.random.default_rng(5)
    tb, th, tu = [], [], []
    for b, L in enumerate(wl.seq_lens):
        for u in np.unique(np.concatenate([[0, L - 1], rng.integers(0, L, size=12)])):
            for h in rng.choice(wl.q_heads, size=3, replace=False):
                tb.append(b); th.append(h); tu.append(u)
    ref = oracle.replay_tokens(wl, layer, q, k, v, g, tb, th, tu)
    G.assert_parity(BF16, _f64(out)[tb, th, tu], ref, "guided layer after a timeout")
