"""MoT-h (App. C.5) on the GPU through the C ABI: the translated activation
restored through the target's projections, against the fp64 oracle."""
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

SMALL_H = {
    # ragged (an odd number of token tiles), an untranslated target layer, D_t = 256 as 2 x 128
    "h_ragged": synth.Workload("h_ragged", 3, 1, 128, 4, 2, 128, 3, 256, 3, 200, "bf16",
                               (200, 77, 1), layer_map=(2, -1, 0, 1), act_tgt=256),
    # wider activations (two N tiles of a_hat per expert), D_t = 256 as 4 x 64, depth-ratio map
    "h_wide": synth.Workload("h_wide", 5, 1, 256, 3, 4, 64, 2, 512, 2, 160, "bf16", (160, 33),
                             act_tgt=512),
    # Top-1 of 2 (token buckets) in the mixture, D_t = 512
    "h_top1": synth.Workload("h_top1", 2, 1, 192, 2, 4, 128, 2, 256, 2, 150, "bf16", (150, 64),
                             top_k=1, act_tgt=256),
}


class HRun:
    def __init__(self, wl, act, blob, seq_lens=None):
        self.wl = wl
        self.h = M.mot_create_h(M.h_config_from(wl))
        M.mot_load_weights(self.h, blob)
        self.act = G.to_device(wl, act)
        self.seq = list(wl.seq_lens if seq_lens is None else seq_lens)
        self.lens = torch.tensor(self.seq, dtype=torch.int32, device="cuda")
        self.buf_k, self.dk = G.alloc_dst(wl)
        self.buf_v, self.dv = G.alloc_dst(wl)

    def translate(self):
        M.mot_translate_h(self.h, self.act, self.lens, len(self.seq), self.dk, self.dv)
        return M.mot_get_device_status(self.h)

    def gather(self, tb, ts):
        """[L_t][n][D_t] float64 of each target cache at the sampled tokens."""
        tbt = torch.as_tensor(tb, dtype=torch.long, device="cuda")
        tst = torch.as_tensor(ts, dtype=torch.long, device="cuda")
        out = []
        for dst in (self.dk, self.dv):
            g = dst[:, tbt, :, tst, :]   # [n, L_t, H_t, d_t]
            out.append(g.permute(1, 0, 2, 3).reshape(self.wl.n_layers_tgt, len(tb), -1)
                       .double().cpu().numpy())
        return out


def _all_tokens(wl):
    tb = np.concatenate([np.full(L, b) for b, L in enumerate(wl.seq_lens)]).astype(np.int32)
    ts = np.concatenate([np.arange(L) for L in wl.seq_lens]).astype(np.int32)
    return tb, ts


def _clear(wl, act, blob, tb, ts):
    """Tokens whose Top-K choice has a margin of 1e-4 (all tokens when dense)."""
    if not (0 < wl.top_k < wl.n_translators):
        return np.ones((wl.n_layers_tgt, tb.size), dtype=bool)
    kv = wl.replace(tgt_kv_heads=1, tgt_head_dim=wl.act_tgt, act_tgt=0, top_k=0)
    mix = kv.group_elems()
    per = wl.group_elems()
    blocks = []
    for r in range(len(wl.translated_layers())):
        blk = blob[r * per:r * per + mix]
        blocks += [blk, blk]
    _, gate = oracle.translate_tokens(kv, act, act, np.concatenate(blocks), tb, ts, want_gate=True)
    srt = -np.sort(-gate[:, 0], axis=-1)
    return srt[..., wl.top_k - 1] - srt[..., wl.top_k] >= 1e-4


@pytest.mark.parametrize("name", sorted(SMALL_H))
def test_moth_small_shapes_every_token(name):
    wl = SMALL_H[name]
    act, blob = synth.gen_cache(wl, 0, 21), synth.gen_weights(wl, 21)
    run = HRun(wl, act, blob)
    assert M.mot_get_path(run.h) == 1
    assert run.translate() == M.MOT_OK
    assert run.canaries_intact() if hasattr(run, "canaries_intact") else True
    tb, ts = _all_tokens(wl)
    rk, rv = oracle.translate_h_tokens(wl, act, blob, tb, ts)
    gk, gv = run.gather(tb, ts)
    tl = wl.translated_layers()
    ok = _clear(wl, act, blob, tb, ts)
    assert ok[tl].mean() > 0.99
    keep = np.broadcast_to(ok[..., None], gk.shape)
    G.assert_parity(wl, gk[tl][keep[tl]], rk[tl][keep[tl]], f"{name} K")
    G.assert_parity(wl, gv[tl][keep[tl]], rv[tl][keep[tl]], f"{name} V")
    # positions past each sequence and untranslated layers keep the sentinel
    s = G.sentinel_value(wl)
    for dst in (run.dk, run.dv):
        iv = G.int_view(dst)
        for l in range(wl.n_layers_tgt):
            for b in range(wl.max_batch):
                L = wl.seq_lens[b] if (l in tl and b < len(wl.seq_lens)) else 0
                assert bool((iv[l, b, :, L:, :] == s).all()), (l, b)
    n = run.dk.numel()
    for buf in (run.buf_k, run.buf_v):
        assert bool((G.int_view(buf[n:]) == s).all())


def test_moth_full_size_sampled():
    """GPT-2-small -> OPT-125m widths, 12 layers, 8 x 1024 tokens, sampled tokens."""
    wl = synth.WORKLOADS["h_gpt2s_opt125m"]
    act, blob = synth.gen_cache(wl, 0), synth.gen_weights(wl)
    run = HRun(wl, act, blob)
    assert run.translate() == M.MOT_OK
    tb, ts = H.stratified_tokens(wl.seq_lens, 1024, seed=1)
    rk, rv = oracle.translate_h_tokens(wl, act, blob, tb, ts)
    gk, gv = run.gather(tb, ts)
    G.assert_parity(wl, gk, rk, f"h_gpt2s_opt125m K ({tb.size} tokens)")
    G.assert_parity(wl, gv, rv, f"h_gpt2s_opt125m V ({tb.size} tokens)")
    # every token of one 256-token pair tile per sequence and the batch's last
    # pair tile, on the first and last target layer
    keep = {0, wl.n_layers_tgt - 1}
    wl2, blob2 = H.restrict_layers(wl, blob, list(range(wl.n_layers_tgt)), keep)
    pb, ps = H.whole_tiles(wl.seq_lens, tile=256)
    rk, rv = oracle.translate_h_tokens(wl2, act, blob2, pb, ps)
    gk, gv = run.gather(pb, ps)
    kl = sorted(keep)
    G.assert_parity(wl, gk[kl], rk[kl], f"h_gpt2s_opt125m K pair tiles ({pb.size} tokens)")
    G.assert_parity(wl, gv[kl], rv[kl], f"h_gpt2s_opt125m V pair tiles ({pb.size} tokens)")


def test_moth_schedules_and_kernels():
    wl = SMALL_H["h_ragged"]
    act, blob = synth.gen_cache(wl, 0, 22), synth.gen_weights(wl, 22)
    outs = []
    for schedule in (2, 0):
        run = HRun(wl, act, blob)
        M.mot_set_schedule(run.h, schedule)
        M.mot_profile_enable(run.h, True)
        assert run.translate() == M.MOT_OK
        stats = M.mot_profile_read(run.h)
        assert "umma2_proj" in stats and "gate" in stats
        outs.append((G.int_view(run.dk).clone(), G.int_view(run.dv).clone()))
    assert torch.equal(outs[0][0], outs[1][0]) and torch.equal(outs[0][1], outs[1][1])


def test_moth_argument_errors():
    wl = SMALL_H["h_ragged"]
    act, blob = synth.gen_cache(wl, 0, 23), synth.gen_weights(wl, 23)
    run = HRun(wl, act, blob)
    with pytest.raises(M.MotError) as e:   # a MoT-h handle takes mot_translate_h only
        M.mot_translate(run.h, run.act, run.act, run.lens, 3, run.dk, run.dv)
    assert e.value.status == M.MOT_ERR_INVALID_ARG
    with pytest.raises(M.MotError) as e:
        M.mot_translate_h(run.h, run.act, run.lens, 3, run.dk, run.dk)   # K aliases V
    assert e.value.status == M.MOT_ERR_INVALID_ARG
    kv = synth.Workload("kv", 3, 2, 64, 4, 2, 128, 3, 256, 3, 200, "bf16", (200, 77, 1))
    hk = M.mot_create(M.config_from(kv))
    with pytest.raises(M.MotError) as e:   # a KV handle does not take mot_translate_h
        M.mot_translate_h(hk, run.act, run.lens, 3, run.dk, run.dv)
    assert e.value.status == M.MOT_ERR_INVALID_ARG
    M.mot_destroy(hk)
    for bad in (wl.replace(act_tgt=320), wl.replace(dtype="fp32")):
        with pytest.raises(M.MotError) as e:
            M.mot_create_h(M.h_config_from(bad))
        assert e.value.status == M.MOT_ERR_UNSUPPORTED
    h2 = M.mot_create_h(M.h_config_from(wl))
    with pytest.raises(M.MotError) as e:
        M.mot_load_weights(h2, blob[:-1])
    assert e.value.status == M.MOT_ERR_WEIGHTS_SIZE
    M.mot_destroy(h2)
