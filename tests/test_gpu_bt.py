"""Backbone translators (App. C.2) inside the gated mixture (Def. 3.1) on the GPU
through the C ABI, against the fp64 oracle."""
import numpy as np
import pytest

import oracle
import synth

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")
if not torch.cuda.is_available():
    pytest.skip("needs a CUDA GPU", allow_module_level=True)

import _helpers as H   # noqa: E402
import _gpu as G   # noqa: E402
M = G.M

W = synth.Workload
SMALL_BT = {
    # GPT-2-small shapes: P = 12 heads (tiles of 10 tokens = 120 rows), ragged, window 1..3
    "bt_p12": W("bt_p12", 6, 12, 64, 6, 12, 64, 2, 0, 2, 50, "bf16", (50, 23),
                bt=(1, 3, 128, 4, 512)),
    # Qwen shapes: P = 2, D_t = 256, Top-1 of 2, a depth-ratio map 6 -> 7, window 2..5
    "bt_p2_top1": W("bt_p2_top1", 6, 2, 64, 7, 2, 128, 2, 0, 2, 300, "bf16", (300, 129),
                    top_k=1, bt=(2, 4, 128, 4, 512)),
    # d_s = 128 (two K blocks), width 64 with heads of 16, FFN 128, E = 3 with Top-2,
    # an empty sequence, window 0..1
    "bt_d64_e3": W("bt_d64_e3", 3, 4, 128, 3, 4, 32, 3, 0, 3, 70, "bf16", (70, 5, 0),
                   top_k=2, bt=(0, 2, 64, 4, 128)),
    # P = 1 (one key: the softmax is 1), FFN 768 (three N tiles), heads of 64, window 3..3
    "bt_p1_ffn768": W("bt_p1_ffn768", 4, 1, 64, 4, 1, 64, 2, 0, 2, 200, "bf16", (200, 131),
                      bt=(3, 1, 128, 2, 768)),
}


class BtRun:
    def __init__(self, wl, sk, sv, blob, seq_lens=None, batch=None):
        self.wl = wl
        cfg, bt = M.bt_config_from(wl)
        self.h = M.mot_create_bt(cfg, bt)
        M.mot_load_weights(self.h, blob)
        self.sk = G.to_device(wl, sk)
        self.sv = G.to_device(wl, sv)
        self.seq = list(wl.seq_lens if seq_lens is None else seq_lens)
        self.batch = len(self.seq) if batch is None else batch
        self.lens = torch.tensor(self.seq, dtype=torch.int32, device="cuda")
        self.buf_k, self.dk = G.alloc_dst(wl)
        self.buf_v, self.dv = G.alloc_dst(wl)

    def translate(self, stream=None):
        M.mot_translate_bt(self.h, self.sk, self.sv, self.lens, self.batch, self.dk, self.dv,
                           stream)
        return M.mot_get_device_status(self.h, stream)

    def gather(self, tb, ts):
        """Window layers at the sampled tokens: [N][2][n][D_t] float64."""
        q, N = self.wl.bt[0], self.wl.bt[1]
        tbt = torch.as_tensor(tb, dtype=torch.long, device="cuda")
        tst = torch.as_tensor(ts, dtype=torch.long, device="cuda")
        out = []
        for dst in (self.dk, self.dv):
            g = dst[q:q + N][:, tbt, :, tst, :]          # [n, N, H_t, d_t]
            out.append(g.permute(1, 0, 2, 3).reshape(N, len(tb), -1).double().cpu().numpy())
        return np.stack(out, axis=1)

    def untouched_outside(self, lens=None):
        """Layers outside the window, padding positions and the canaries keep the sentinel."""
        wl, s = self.wl, G.sentinel_value(self.wl)
        lens = self.seq if lens is None else lens
        win = set(wl.bt_window)
        n = self.dk.numel()
        for buf, dst in ((self.buf_k, self.dk), (self.buf_v, self.dv)):
            if not bool((G.int_view(buf[n:]) == s).all()):
                return False
            iv = G.int_view(dst)
            for l in range(wl.n_layers_tgt):
                for b in range(wl.max_batch):
                    L = lens[b] if (l in win and b < self.batch) else 0
                    L = max(0, min(L, wl.max_seq))
                    if not bool((iv[l, b, :, L:, :] == s).all()):
                        return False
        return True


def _inputs(wl, seed=0):
    return synth.gen_cache(wl, 0, seed), synth.gen_cache(wl, 1, seed), synth.gen_weights(wl, seed)


def _all_tokens(seq):
    tb = np.concatenate([np.full(L, b) for b, L in enumerate(seq) if L > 0]).astype(np.int32)
    ts = np.concatenate([np.arange(L) for L in seq if L > 0]).astype(np.int32)
    return tb, ts


def _clear(wl, gate):
    """[2][n] tokens whose Top-K choice has a margin of 1e-4 in the oracle's gate
    (near-ties may legitimately select differently in fp32)."""
    if not (0 < wl.top_k < wl.n_translators):
        return np.ones(gate.shape[:2], dtype=bool)
    srt = -np.sort(-gate, axis=-1)
    return srt[..., wl.top_k - 1] - srt[..., wl.top_k] >= 1e-4


def _dense_gate(wl, sk, sv, blob, tb, ts):
    _, g = oracle.bt_tokens(wl.replace(top_k=0), sk, sv, blob, tb, ts, want_gate=True)
    return g


@pytest.mark.parametrize("name", sorted(SMALL_BT))
def test_bt_matches_oracle_on_every_token(name):
    wl = SMALL_BT[name]
    sk, sv, blob = _inputs(wl)
    run = BtRun(wl, sk, sv, blob)
    assert run.translate() == M.MOT_OK
    tb, ts = _all_tokens(wl.seq_lens)
    ref = oracle.bt_tokens(wl, sk, sv, blob, tb, ts)
    got = run.gather(tb, ts)
    clear = _clear(wl, _dense_gate(wl, sk, sv, blob, tb, ts))
    assert clear.mean() > 0.9
    for X in range(2):
        G.assert_parity(wl, got[:, X][:, clear[X]], ref[:, X][:, clear[X]], f"{name} X={X}")
    assert run.untouched_outside()


def test_bt_full_size_sampled_tokens():
    """GPT-2-small -> OPT-125m backbone workload at full size (8 x 1024 tokens),
    in the launch configuration the benchmark times, on sampled tokens."""
    wl = synth.WORKLOADS["bt_gpt2s_opt125m"].replace(top_k=0)   # dense gate: every backbone
    sk, sv, blob = _inputs(wl)
    run = BtRun(wl, sk, sv, blob)
    assert run.translate() == M.MOT_OK
    # a stratified sample of the batch, plus 40 consecutive tokens per sequence
    # (whole 10-token row tiles of P = 12 source-head rows) and the batch's end
    tb, ts = H.stratified_tokens(wl.seq_lens, 1024, seed=3, tile=10)
    pb, ps = H.whole_tiles(wl.seq_lens, tile=40, seed=5)
    tb, ts = np.concatenate([tb, pb]), np.concatenate([ts, ps])
    ref = oracle.bt_tokens(wl, sk, sv, blob, tb, ts)
    got = run.gather(tb, ts)
    G.assert_parity(wl, got, ref, f"bt_gpt2s_opt125m ({tb.size} tokens)")


def test_bt_full_size_top1_routed_sampled_tokens():
    """The GPT-2-small -> OPT-125m backbone workload at full size with the
    paper's default Top-1 of 2 backbones on token buckets."""
    wl = synth.WORKLOADS["bt_gpt2s_opt125m"]
    assert wl.top_k == 1
    sk, sv, blob = _inputs(wl)
    run = BtRun(wl, sk, sv, blob)
    assert M.mot_get_routing(run.h) == 1
    assert run.translate() == M.MOT_OK
    assert run.untouched_outside()
    tb, ts = H.stratified_tokens(wl.seq_lens, 512, seed=6, tile=10)
    ref = oracle.bt_tokens(wl, sk, sv, blob, tb, ts)
    dense = _dense_gate(wl, sk, sv, blob, tb, ts)
    clear = _clear(wl, dense)
    assert clear.mean() > 0.99
    got = run.gather(tb, ts)
    for X in range(2):
        G.assert_parity(wl, got[:, X][:, clear[X]], ref[:, X][:, clear[X]], f"Top-1 X={X}")


def test_bt_qwen_shapes_sampled_tokens():
    wl = synth.WORKLOADS["bt_qwen05_qwen15"].replace(max_batch=2, max_seq=1024,
                                                     seq_lens=(1024, 700))
    sk, sv, blob = _inputs(wl, 1)
    run = BtRun(wl, sk, sv, blob)
    assert run.translate() == M.MOT_OK
    tb, ts = H.stratified_tokens(wl.seq_lens, 256, seed=4, tile=64)
    ref = oracle.bt_tokens(wl, sk, sv, blob, tb, ts)
    clear = _clear(wl, _dense_gate(wl, sk, sv, blob, tb, ts))   # Top-1: skip near-ties
    got = run.gather(tb, ts)
    for X in range(2):
        G.assert_parity(wl, got[:, X][:, clear[X]], ref[:, X][:, clear[X]],
                        f"bt_qwen05_qwen15 X={X}")


def test_bt_one_hot_gate_is_one_backbone_and_deterministic():
    """Wg = 0, bg = 9984 e_1: every token uses backbone 1 alone; two runs agree bit for bit."""
    wl = SMALL_BT["bt_p12"]
    sk, sv, blob = _inputs(wl, 2)
    blob = blob.copy()
    for (x, name, m, r, off, n, _, _) in synth.bt_blob_offsets(wl):
        if name == "wg":
            blob[off:off + n] = 0
        elif name == "bg":
            blob[off:off + n] = np.array([0, 0x461C], dtype=np.uint16)   # 0 and 9984 (bf16)
    run = BtRun(wl, sk, sv, blob)
    assert run.translate() == M.MOT_OK
    first = [run.dk.clone(), run.dv.clone()]
    tb, ts = _all_tokens(wl.seq_lens)
    ref = oracle.bt_tokens(wl, sk, sv, blob, tb, ts)
    G.assert_parity(wl, run.gather(tb, ts), ref, "one-hot")
    assert run.translate() == M.MOT_OK
    assert torch.equal(G.int_view(first[0]), G.int_view(run.dk))
    assert torch.equal(G.int_view(first[1]), G.int_view(run.dv))


def test_bt_batch_prefix_and_length_clamp():
    """batch < max_batch leaves later entries alone; a length above max_seq is
    clamped and reported (MOT_ERR_SEQ_LEN)."""
    wl = SMALL_BT["bt_p12"]
    sk, sv, blob = _inputs(wl, 5)
    run = BtRun(wl, sk, sv, blob, seq_lens=[50, 40], batch=1)
    assert run.translate() == M.MOT_OK
    assert run.untouched_outside(lens=[50, 0])
    run2 = BtRun(wl, sk, sv, blob, seq_lens=[999, 7])
    assert run2.translate() == M.MOT_ERR_SEQ_LEN
    tb, ts = _all_tokens([50, 7])
    ref = oracle.bt_tokens(wl, sk, sv, blob, tb, ts)
    G.assert_parity(wl, run2.gather(tb, ts), ref, "clamped")
    assert run2.untouched_outside(lens=[50, 7])


@pytest.mark.parametrize("routing", [1, 0])
def test_bt_launch_sequence_and_profile(routing):
    """Dense: the gate, then 7 launches per window slot. Top-1 routing (token
    buckets, the default for a Top-1 handle): the gate and the route kernel, then
    per slot the bucket tokens' source rows are packed before the 7 stages."""
    wl = SMALL_BT["bt_p2_top1"]
    sk, sv, blob = _inputs(wl)
    run = BtRun(wl, sk, sv, blob)
    assert M.mot_get_routing(run.h) == 1   # the default for top_k = 1
    M.mot_set_routing(run.h, routing)
    M.mot_profile_enable(run.h, True)
    c0 = M.mot_get_launch_count(run.h)
    assert run.translate() == M.MOT_OK
    N, d_f = wl.bt[1], wl.bt[4]
    fused = d_f % 128 == 0   # FFN1 + GELU + FFN2 in one kernel
    per_slot = (7 if fused else 8) + (1 if routing else 0)
    assert M.mot_get_launch_count(run.h) - c0 == 1 + routing + per_slot * N
    prof = M.mot_profile_read(run.h)
    ffn = {"bt_ffn_fused"} if fused else {"bt_ffn1_gelu", "bt_ffn2_residual_ln"}
    routed = {"bt_route", "bt_pack"} if routing else set()
    assert set(prof) == {"bt_gate", "bt_in_ln_gelu", "bt_q", "bt_kv", "bt_attn",
                         "bt_o_residual_ln", "bt_out_gelu_combine"} | ffn | routed
    assert prof["bt_gate"][0] == 1 and prof["bt_q"][0] == N


ROUTED = {
    "bt_p2_top1": SMALL_BT["bt_p2_top1"],
    # P = 12 (120-row tiles of 10 tokens), Top-1 of 3, ragged with an empty sequence
    "bt_p12_top1": W("bt_p12_top1", 6, 12, 64, 6, 12, 64, 3, 0, 3, 50, "bf16", (50, 23, 0),
                     top_k=1, bt=(1, 3, 128, 4, 512)),
    # FFN 768 (unfused FFN, three N tiles), P = 1, Top-1 of 2
    "bt_p1_top1": W("bt_p1_top1", 4, 1, 64, 4, 1, 64, 2, 0, 2, 200, "bf16", (200, 131),
                    top_k=1, bt=(3, 1, 128, 2, 768)),
}


@pytest.mark.parametrize("name", sorted(ROUTED))
def test_bt_top1_token_buckets_equal_dense_and_oracle(name):
    """Top-1 of E (Def. 3.1 with backbone experts): running each backbone only on
    the tokens that chose it (token buckets) gives bit for bit the dense result
    (every backbone on every token, the unchosen weighted by zero), and both
    match the oracle; the bucket sizes are the oracle's choice counts."""
    wl = ROUTED[name]
    sk, sv, blob = _inputs(wl, 8)
    runs = []
    for routing in (1, 0):
        run = BtRun(wl, sk, sv, blob)
        M.mot_set_routing(run.h, routing)
        assert run.translate() == M.MOT_OK
        assert run.untouched_outside()
        runs.append(run)
    assert torch.equal(G.int_view(runs[0].dk), G.int_view(runs[1].dk))
    assert torch.equal(G.int_view(runs[0].dv), G.int_view(runs[1].dv))
    tb, ts = _all_tokens(wl.seq_lens)
    ref, gate = oracle.bt_tokens(wl, sk, sv, blob, tb, ts, want_gate=True)
    got = runs[0].gather(tb, ts)
    dense = _dense_gate(wl, sk, sv, blob, tb, ts)
    clear = _clear(wl, dense)
    for X in range(2):
        G.assert_parity(wl, got[:, X][:, clear[X]], ref[:, X][:, clear[X]], f"{name} X={X}")
    counts = M.mot_get_expert_counts(runs[0].h, 2, wl.n_translators)
    want = np.stack([(gate[X] > 0).sum(axis=0) for X in range(2)])
    assert (np.abs(counts - want) <= (~clear).sum(axis=1)[:, None]).all(), (counts, want)
    assert counts.sum() == 2 * tb.size


def test_bt_argument_errors():
    wl = SMALL_BT["bt_p12"]
    cfg, bt = M.bt_config_from(wl)
    for bad in [(5, 2, 128, 4, 512), (0, 0, 128, 4, 512), (0, 2, 128, 3, 512)]:
        with pytest.raises(M.MotError) as e:
            M.mot_create_bt(cfg, M.mot_bt_config(*bad))
        assert e.value.status == M.MOT_ERR_INVALID_ARG
    for bad in [(0, 2, 96, 4, 512), (0, 2, 128, 4, 100)]:   # unsupported width / FFN
        with pytest.raises(M.MotError) as e:
            M.mot_create_bt(cfg, M.mot_bt_config(*bad))
        assert e.value.status == M.MOT_ERR_UNSUPPORTED
    with pytest.raises(M.MotError) as e:
        M.mot_create_bt(M.config_from(wl.replace(dtype="fp32")), bt)
    assert e.value.status == M.MOT_ERR_UNSUPPORTED
    sk, sv, blob = _inputs(wl)
    h = M.mot_create_bt(cfg, bt)
    with pytest.raises(M.MotError) as e:
        M.mot_load_weights(h, blob[:-1])
    assert e.value.status == M.MOT_ERR_WEIGHTS_SIZE
    run = BtRun(wl, sk, sv, blob)
    with pytest.raises(M.MotError) as e:   # a backbone handle takes mot_translate_bt only
        M.mot_translate(run.h, run.sk, run.sv, run.lens, 2, run.dk, run.dv)
    assert e.value.status == M.MOT_ERR_INVALID_ARG
    with pytest.raises(M.MotError) as e:   # dst aliasing src
        M.mot_translate_bt(run.h, run.sk, run.sv, run.lens, 2, run.sk, run.dv)
    assert e.value.status == M.MOT_ERR_INVALID_ARG
