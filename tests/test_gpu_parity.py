"""CUDA path vs the fp64 oracle, element by element, through the C ABI."""
import numpy as np
import pytest

import oracle
import synth
import _helpers as H

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")
if not torch.cuda.is_available():
    pytest.skip("needs a CUDA GPU", allow_module_level=True)

import _gpu as G   # noqa: E402
M = G.M


def inputs(wl, seed=0):
    return synth.gen_cache(wl, 0, seed), synth.gen_cache(wl, 1, seed), synth.gen_weights(wl, seed)


def full_check(wl, run, sk, sv, blob, label):
    """Every element against oracle.translate_full; untouched positions keep the sentinel."""
    assert run.canaries_intact(), f"{label}: wrote past the end of dst"
    assert run.padding_untouched(), f"{label}: wrote a position it must not touch"
    rk, rv = oracle.translate_full(wl, sk, sv, blob, run.seq[:run.batch])
    gk, gv = run.dst_f64()
    mask = G.translated_mask_full(wl, run.seq, run.batch)
    mk = G.assert_parity(wl, gk[mask], rk[mask], label + " K")
    mv = G.assert_parity(wl, gv[mask], rv[mask], label + " V")
    return mk, mv


# ---------------------------------------------------------------- small shapes, every element

SMALL = {
    # tensor-core path: ragged tails, several tiles, D_s != D_t, a -1 in the map, unused batch slot
    "umma_ragged": synth.Workload("umma_ragged", 3, 2, 64, 4, 2, 128, 2, 256, 4, 300, "bf16",
                                  (300, 129, 1), layer_map=(2, -1, 0, 1)),
    # tensor-core path, E = 3, 128-dim source heads, depth-ratio map 5 -> 3
    "umma_e3": synth.Workload("umma_e3", 5, 1, 128, 3, 4, 64, 3, 512, 2, 200, "bf16", (200, 77)),
    # SIMT path (head dims outside the tensor-core tiling), bf16
    "simt_bf16": synth.Workload("simt_bf16", 2, 3, 16, 2, 5, 8, 3, 40, 2, 70, "bf16", (70, 33)),
    # SIMT path, fp32, odd sizes
    "simt_fp32": synth.Workload("simt_fp32", 3, 2, 12, 2, 3, 10, 2, 50, 3, 90, "fp32",
                                (90, 0, 65), layer_map=(2, 0)),
    # single translator (E = 1) on the tensor-core path
    "umma_e1": synth.Workload("umma_e1", 2, 4, 64, 2, 2, 128, 1, 512, 1, 256, "bf16", (256,)),
    # D_t = 512 (two CTA pairs per cluster): ragged, an odd tile count (the last
    # pair tile has one live half), a -1 in the map, E = 3 (6 hidden chunks)
    "umma_wide": synth.Workload("umma_wide", 3, 4, 64, 4, 4, 128, 3, 256, 3, 300, "bf16",
                                (300, 129, 1), layer_map=(2, -1, 0, 1)),
    # D_t = 512, D_s = 512 (8 K blocks), E = 1, H = 768 (6 chunks)
    "umma_wide_e1": synth.Workload("umma_wide_e1", 2, 4, 128, 2, 4, 128, 1, 768, 2, 256, "bf16",
                                   (256, 200)),
}


def onchip_supported(wl):
    """Shapes the on-chip schedule (3) takes: D_s <= 128, D_t = 256, bf16 tensor-core path."""
    d_s, d_t = wl.src_kv_heads * wl.src_head_dim, wl.tgt_kv_heads * wl.tgt_head_dim
    return (wl.dtype == "bf16" and d_s <= 128 and d_t == 256 and wl.hidden % 256 == 0
            and wl.src_head_dim % 64 == 0 and wl.tgt_head_dim % 32 == 0)


def wide_supported(wl):
    """Shapes the on-chip schedule on clusters of two CTA pairs (4) takes: D_t = 512."""
    d_t = wl.tgt_kv_heads * wl.tgt_head_dim
    return (wl.dtype == "bf16" and d_t == 512 and wl.hidden % 256 == 0
            and wl.src_head_dim % 64 == 0 and wl.tgt_head_dim % 32 == 0)


def schedule_supported(wl, schedule):
    if schedule == 3:
        return onchip_supported(wl)
    if schedule == 4:
        return wide_supported(wl)
    return True


@pytest.mark.parametrize("schedule", [4, 3, 2, 1, 0])
@pytest.mark.parametrize("name", sorted(SMALL))
def test_small_shapes_every_element(name, schedule):
    wl = SMALL[name]
    if schedule != 2 and not name.startswith("umma"):
        pytest.skip("the schedule only applies to the tensor-core path")
    if not schedule_supported(wl, schedule):
        pytest.skip("the schedule does not take this shape")
    sk, sv, blob = inputs(wl, seed=1)
    run = G.Run(wl, sk, sv, blob)
    expect_path = 1 if name.startswith("umma") else 0
    assert M.mot_get_path(run.h) == expect_path
    M.mot_set_schedule(run.h, schedule)
    assert run.translate() == M.MOT_OK
    full_check(wl, run, sk, sv, blob, name)


@pytest.mark.parametrize("other", [1, 2, 3, 4])
@pytest.mark.parametrize("name", ["umma_ragged", "umma_e3", "umma_wide", "umma_wide_e1",
                                  "gpt2s_opt125m", "qwen7_long", "qwen05_qwen15", "gpt2m_qwen7"])
def test_launch_schedules_are_bit_identical(name, other):
    """Every launch schedule runs the same per-tile arithmetic in the same order."""
    wl = SMALL.get(name) or synth.WORKLOADS[name]
    if not schedule_supported(wl, other):
        pytest.skip("the schedule does not take this shape")
    sk, sv, blob = inputs(wl, seed=3)
    a = G.Run(wl, sk, sv, blob)
    b = G.Run(wl, sk, sv, blob)
    M.mot_set_schedule(a.h, 0)
    M.mot_set_schedule(b.h, other)
    assert a.translate() == M.MOT_OK and b.translate() == M.MOT_OK
    assert torch.equal(G.int_view(a.dk), G.int_view(b.dk))
    assert torch.equal(G.int_view(a.dv), G.int_view(b.dv))


def test_tiny_fp32_workload_every_element():
    """The fp32 GPT-2-small -> OPT-125m-shaped workload (4 layers, seq 64, E=2), in full."""
    wl = synth.WORKLOADS["tiny_fp32"]
    sk, sv, blob = inputs(wl)
    run = G.Run(wl, sk, sv, blob)
    assert run.translate() == M.MOT_OK
    full_check(wl, run, sk, sv, blob, wl.name)


# ---------------------------------------------------------------- full-size workloads, sampled

# tokens sampled over the whole batch per workload (the oracle's cost per token
# grows with D_s * H * E: the two largest get fewer)
FULL_SIZE_SAMPLE = {"gpt2s_opt125m": 1024, "qwen05_qwen15": 1024, "gpt2m_qwen7": 256,
                    "qwen7_long": 256}


@pytest.mark.parametrize("name", sorted(FULL_SIZE_SAMPLE))
def test_full_size_workload_sampled(name):
    """The workload at full size in the benchmark's launch configuration, against
    the oracle on (a) a stratified token sample over every sequence (ends and
    128-token tile boundaries included), on every translated layer, and (b)
    every token of one 256-token pair tile per sequence plus the last pair tile
    of the batch (the persistent schedule's last wave), on the first and the
    last target layer. Every untouched position must still hold the sentinel."""
    wl = synth.WORKLOADS[name]
    sk, sv, blob = inputs(wl)
    run = G.Run(wl, sk, sv, blob)
    assert run.translate() == M.MOT_OK
    assert run.canaries_intact() and run.padding_untouched()
    tb, ts = H.stratified_tokens(wl.seq_lens, FULL_SIZE_SAMPLE[name], seed=1)
    ref = oracle.translate_tokens(wl, sk, sv, blob, tb, ts)
    got = run.gather(tb, ts)
    tl = wl.translated_layers()
    m = G.assert_parity(wl, got[tl], ref[tl], f"{name} stratified ({tb.size} tokens)")
    print(name, "stratified", tb.size, m)
    lm = M.mot_get_layer_map(run.h)
    keep = {tl[0], tl[-1]}
    wl2, blob2 = H.restrict_layers(wl, blob, lm, keep)
    pb, ps = H.whole_tiles(wl.seq_lens, tile=256)
    ref2 = oracle.translate_tokens(wl2, sk, sv, blob2, pb, ps)
    got2 = run.gather(pb, ps)
    kl = sorted(keep)
    m2 = G.assert_parity(wl, got2[kl], ref2[kl], f"{name} whole pair tiles ({pb.size} tokens)")
    print(name, "pair tiles", pb.size, m2)


# ---------------------------------------------------------------- invariants on the GPU

def _identity_blob(wl):
    D = wl.d_src

    def fn(l, x):
        tr = [H.signed_perm_translator(D, wl.hidden, np.arange(D), np.arange(D))
              for _ in range(wl.n_translators)]
        return dict(Wg=np.zeros((wl.n_translators, D)), bg=np.zeros(wl.n_translators),
                    W1=[t[0] for t in tr], b1=[t[1] for t in tr], W2=[t[2] for t in tr],
                    b2=[t[3] for t in tr])
    return H.make_blob(wl, fn)


def test_identity_translator_copies_the_cache():
    """W1=[I;-I], W2=[I,-I]: each translated layer is the mapped source layer,
    re-headed from 4x64 to 2x128 (bf16 rounding of the hidden layer aside)."""
    wl = synth.Workload("ident", 3, 4, 64, 4, 2, 128, 2, 512, 2, 160, "bf16", (160, 40))
    sk, sv, _ = inputs(wl, seed=2)
    blob = _identity_blob(wl)
    run = G.Run(wl, sk, sv, blob)
    assert M.mot_get_path(run.h) == 1
    assert run.translate() == M.MOT_OK
    gk, gv = run.dst_f64()
    lm = oracle.depth_ratio_map(3, 4)
    assert M.mot_get_layer_map(run.h) == lm
    for l in range(4):
        for src, got in ((sk, gk), (sv, gv)):
            for b, L in enumerate(wl.seq_lens):
                z = H.storage_to_f64(wl, src[lm[l], b, :, :L, :]).transpose(1, 0, 2).reshape(L, -1)
                y = got[l, b, :, :L, :].transpose(1, 0, 2).reshape(L, -1)
                # hidden activations are rounded to bf16 before the second GEMM
                np.testing.assert_allclose(y, z, rtol=1e-2, atol=2e-2)


def test_one_hot_gate_equals_single_translator_run():
    """Proof of Prop. 3.1 on the GPU: a one-hot gate over E=3 gives the E=1 result."""
    wl3 = synth.Workload("oh3", 2, 2, 64, 2, 2, 128, 3, 256, 1, 256, "bf16", (256,))
    wl1 = wl3.replace(n_translators=1)
    sk, sv, blob = inputs(wl3, seed=4)
    grp = H.split_blob(wl3, blob)
    m0 = 2

    def onehot(l, x):
        g = dict(grp[(l, x)])
        g["Wg"] = np.zeros_like(g["Wg"])
        g["bg"] = np.array([0.0, 0.0, 1e4])
        return g

    def single(l, x):
        g = grp[(l, x)]
        return dict(Wg=np.zeros((1, wl3.d_src)), bg=np.zeros(1), W1=[g["W1"][m0]], b1=[g["b1"][m0]],
                    W2=[g["W2"][m0]], b2=[g["b2"][m0]])
    r3 = G.Run(wl3, sk, sv, H.make_blob(wl3, onehot))
    r1 = G.Run(wl1, sk, sv, H.make_blob(wl1, single))
    assert r3.translate() == M.MOT_OK and r1.translate() == M.MOT_OK
    a, b = r3.dst_f64(), r1.dst_f64()
    for x in (0, 1):
        np.testing.assert_array_equal(a[x], b[x])


def test_prefix_consistency_and_unused_batch_slots():
    """Shorter sequences give bit-identical values on their prefix; batch slots
    beyond `batch` and positions past each length are untouched."""
    wl = SMALL["umma_ragged"]
    sk, sv, blob = inputs(wl, seed=5)
    full = G.Run(wl, sk, sv, blob)
    assert full.translate() == M.MOT_OK
    short = G.Run(wl, sk, sv, blob, seq_lens=(131, 5, 1))
    assert short.translate() == M.MOT_OK
    assert short.padding_untouched() and short.canaries_intact()
    for a, b in ((full.dk, short.dk), (full.dv, short.dv)):
        for bb, L in enumerate((131, 5, 1)):
            assert torch.equal(G.int_view(a[:, bb, :, :L]), G.int_view(b[:, bb, :, :L]))


def test_zero_length_batch_and_batch_zero():
    wl = SMALL["umma_ragged"]
    sk, sv, blob = inputs(wl, seed=6)
    run = G.Run(wl, sk, sv, blob, seq_lens=(0, 0, 0))
    assert run.translate() == M.MOT_OK
    assert run.padding_untouched()
    run2 = G.Run(wl, sk, sv, blob, seq_lens=(5,), batch=0)
    assert run2.translate() == M.MOT_OK
    assert run2.padding_untouched(lens=[0, 0, 0, 0])


def test_seq_len_out_of_range_is_clamped_and_reported():
    wl = SMALL["umma_ragged"]
    sk, sv, blob = inputs(wl, seed=7)
    bad = G.Run(wl, sk, sv, blob, seq_lens=(wl.max_seq + 50, -3, 10))
    assert bad.translate() == M.MOT_ERR_SEQ_LEN
    assert M.mot_get_device_status(bad.h) == M.MOT_OK     # reading clears the word
    good = G.Run(wl, sk, sv, blob, seq_lens=(wl.max_seq, 0, 10))
    assert good.translate() == M.MOT_OK
    assert torch.equal(G.int_view(bad.dk), G.int_view(good.dk))
    assert torch.equal(G.int_view(bad.dv), G.int_view(good.dv))


HOST_CASES = {
    "ragged": (SMALL["umma_ragged"], None),
    "uniform_partial_batch": (SMALL["umma_ragged"].replace(seq_lens=(200, 200)), None),
    "uniform_full_batch": (SMALL["umma_e3"].replace(seq_lens=(200, 200)), None),
    # 10 translated layers: chunks of 1, 2, 4, 2 and 1 layers
    "many_layers": (synth.Workload("host_many", 9, 2, 64, 10, 2, 128, 2, 256, 2, 160, "bf16",
                                   (160, 77)), None),
}


@pytest.mark.parametrize("case", sorted(HOST_CASES))
def test_host_buffer_entry_point_matches_device_entry_point(case):
    """The pipelined host-buffer path copies only real tokens (one strided copy per
    run of layers when lengths are equal, per batch entry when ragged) and must
    give the device entry point's bytes exactly, leaving every other position."""
    wl, _ = HOST_CASES[case]
    sk, sv, blob = inputs(wl, seed=8)
    run = G.Run(wl, sk, sv, blob)
    assert run.translate() == M.MOT_OK
    dt = torch.int16 if wl.dtype == "bf16" else torch.int32
    hk = torch.from_numpy(sk.view(np.int16)).pin_memory()
    hv = torch.from_numpy(sv.view(np.int16)).pin_memory()
    ok = torch.full(wl.dst_shape(), G.sentinel_value(wl), dtype=dt).pin_memory()
    ov = torch.full(wl.dst_shape(), G.sentinel_value(wl), dtype=dt).pin_memory()
    lens = np.asarray(wl.seq_lens, dtype=np.int32)
    st = torch.cuda.current_stream()
    M.mot_translate_host(run.h, hk, hv, lens, len(lens), ok, ov, st)
    st.synchronize()
    assert torch.equal(ok, G.int_view(run.dk).cpu())
    assert torch.equal(ov, G.int_view(run.dv).cpu())
    with pytest.raises(M.MotError) as e:
        M.mot_translate_host(run.h, hk, hv, np.asarray([wl.max_seq + 1], np.int32), 1, ok, ov, st)
    assert e.value.status == M.MOT_ERR_SEQ_LEN


def test_argument_errors_with_a_live_handle():
    wl = SMALL["umma_ragged"]
    sk, sv, blob = inputs(wl, seed=9)
    h = M.mot_create(M.config_from(wl))
    with pytest.raises(M.MotError) as e:
        M.mot_load_weights(h, blob[:-1])
    assert e.value.status == M.MOT_ERR_WEIGHTS_SIZE
    k, v = G.to_device(wl, sk), G.to_device(wl, sv)
    _, dk = G.alloc_dst(wl)
    _, dv = G.alloc_dst(wl)
    lens = torch.tensor(wl.seq_lens, dtype=torch.int32, device="cuda")
    with pytest.raises(M.MotError) as e:
        M.mot_translate(h, k, v, lens, 3, dk, dv)
    assert e.value.status == M.MOT_ERR_NO_WEIGHTS
    M.mot_load_weights(h, blob)
    for args, why in [((k.data_ptr() + 2, v, lens, 3, dk, dv), "misaligned"),
                      ((k, v, lens, 5, dk, dv), "batch > max_batch"),
                      ((k, v, lens, -1, dk, dv), "negative batch"),
                      ((k, v, lens, 3, dk, dk), "dst_k aliases dst_v"),
                      ((k, v, None, 3, dk, dv), "NULL seq_lens")]:
        with pytest.raises(M.MotError) as e:
            M.mot_translate(h, *args)
        assert e.value.status == M.MOT_ERR_INVALID_ARG, why
    M.mot_destroy(h)


@pytest.mark.parametrize("schedule,kernels", [
    (3, {"prep_tiles", "gate", "umma2_onchip_translate"}),
    (2, {"prep_tiles", "gate", "umma2_gemm1_gelu_gate", "umma2_gemm2_combine_store"}),
    (1, {"prep_tiles", "gate", "umma_fused_translate"}),
    (0, {"prep_tiles", "gate", "umma_gemm1_gelu_gate", "umma_gemm2_combine_store"})])
def test_profile_and_launch_count(schedule, kernels):
    wl = SMALL["umma_ragged"]
    sk, sv, blob = inputs(wl, seed=10)
    run = G.Run(wl, sk, sv, blob)
    assert M.mot_get_schedule(run.h) == 3   # the default where the on-chip schedule applies
    M.mot_set_schedule(run.h, schedule)
    n0 = M.mot_get_launch_count(run.h)
    M.mot_profile_enable(run.h, True)
    assert run.translate() == M.MOT_OK
    stats = M.mot_profile_read(run.h)
    assert set(stats) == kernels
    assert all(v[0] >= 1 and v[1] > 0 for v in stats.values())
    assert M.mot_get_launch_count(run.h) - n0 == sum(v[0] for v in stats.values())


@pytest.mark.parametrize("lead", [8, 16])
def test_target_cache_aligned_to_16_but_not_32_bytes(lead):
    """The output stores take 32-byte vectors only where the target cache allows."""
    wl = SMALL["umma_ragged"]
    sk, sv, blob = inputs(wl, seed=12)
    run = G.Run(wl, sk, sv, blob, dst_lead=lead)
    assert run.dk.data_ptr() % 32 == (16 if lead == 8 else 0)
    for schedule in (3, 2):
        M.mot_set_schedule(run.h, schedule)
        assert run.translate() == M.MOT_OK
        full_check(wl, run, sk, sv, blob, f"lead {lead} schedule {schedule}")


def test_onchip_schedule_is_refused_where_unsupported():
    """D_t = 256 with D_s = 256: the default stays 2, asking for 3 (D_s <= 128) or
    4 (D_t = 512) is MOT_ERR_UNSUPPORTED, and 5 is not a schedule."""
    wl = SMALL["umma_e1"]
    sk, sv, blob = inputs(wl, seed=11)
    run = G.Run(wl, sk, sv, blob)
    assert M.mot_get_schedule(run.h) == 2
    for sched in (3, 4):
        with pytest.raises(M.MotError) as e:
            M.mot_set_schedule(run.h, sched)
        assert e.value.status == M.MOT_ERR_UNSUPPORTED
    assert M.mot_get_schedule(run.h) == 2
    with pytest.raises(M.MotError) as e:
        M.mot_set_schedule(run.h, 5)
    assert e.value.status == M.MOT_ERR_INVALID_ARG


# ---------------------------------------------------------------- Top-K routing (Def. 3.1)

TOPK = {
    # the paper's default (Top-K, N_Tr) = (1, 2), tensor-core path
    "umma_top1_of2": synth.Workload("umma_top1_of2", 2, 2, 64, 3, 2, 128, 2, 256, 2, 200, "bf16",
                                    (200, 61), top_k=1),
    # (2, 4), tensor-core path
    "umma_top2_of4": synth.Workload("umma_top2_of4", 2, 2, 64, 2, 2, 128, 4, 256, 2, 160, "bf16",
                                    (160, 33), top_k=2),
    # SIMT fp32 path, Top-3 of 5
    "simt_fp32_top3_of5": synth.Workload("simt_fp32_top3_of5", 2, 2, 12, 2, 3, 10, 5, 30, 2, 50,
                                         "fp32", (50, 17), top_k=3),
}


@pytest.mark.parametrize("name", sorted(TOPK))
def test_topk_routing_against_oracle(name):
    """Top-K keeps the K largest gate scores and renormalises over them. Where
    the K-th and (K+1)-th scores are within 1e-4, fp32 and fp64 may keep
    different experts (both valid): such tokens are excluded, and must be rare."""
    wl = TOPK[name]
    sk, sv, blob = inputs(wl, seed=12)
    run = G.Run(wl, sk, sv, blob)
    assert run.translate() == M.MOT_OK
    assert run.canaries_intact() and run.padding_untouched()
    tb = np.concatenate([np.full(L, b) for b, L in enumerate(wl.seq_lens)]).astype(np.int32)
    ts = np.concatenate([np.arange(L) for L in wl.seq_lens]).astype(np.int32)
    ref, _ = oracle.translate_tokens(wl, sk, sv, blob, tb, ts, want_gate=True)
    _, dense = oracle.translate_tokens(wl.replace(top_k=0), sk, sv, blob, tb, ts, want_gate=True)
    srt = -np.sort(-dense, axis=-1)                       # [L_t][2][n][E], descending
    margin = srt[..., wl.top_k - 1] - srt[..., wl.top_k]  # [L_t][2][n]
    ok = margin >= 1e-4
    tl = wl.translated_layers()
    assert ok[tl].mean() > 0.99
    got = run.gather(tb, ts)
    keep = np.broadcast_to(ok[..., None], got.shape)
    G.assert_parity(wl, got[tl][keep[tl]], ref[tl][keep[tl]], name)


# ---------------------------------------------------------------- Top-K routing with token buckets

TOPK_ROUTED = {
    # two 256-column tiles per expert (H = 512) and per output (D_t = 512), D_s = 256,
    # ragged lengths (odd bucket sizes: padded pair tiles), an untranslated target layer
    "routed_top2_of4": synth.Workload("routed_top2_of4", 3, 4, 64, 3, 4, 128, 4, 512, 3, 300,
                                      "bf16", (300, 129, 7), top_k=2, layer_map=(2, -1, 0)),
    # Top-1 of 8 on the on-chip shapes (D_s = 128, D_t = 256)
    "routed_top1_of8": synth.Workload("routed_top1_of8", 2, 2, 64, 2, 2, 128, 8, 256, 2, 400,
                                      "bf16", (400, 250), top_k=1),
}
ROUTED_ALL = {**{k: v for k, v in TOPK.items() if k.startswith("umma")}, **TOPK_ROUTED}


def _all_tokens(wl):
    tb = np.concatenate([np.full(L, b) for b, L in enumerate(wl.seq_lens)]).astype(np.int32)
    ts = np.concatenate([np.arange(L) for L in wl.seq_lens]).astype(np.int32)
    return tb, ts


def _clear_choice(wl, sk, sv, blob, tb, ts):
    """Tokens whose K-th and (K+1)-th dense gate scores differ by at least 1e-4
    (fp32 and fp64 then keep the same translators)."""
    _, dense = oracle.translate_tokens(wl.replace(top_k=0), sk, sv, blob, tb, ts, want_gate=True)
    srt = -np.sort(-dense, axis=-1)
    return srt[..., wl.top_k - 1] - srt[..., wl.top_k] >= 1e-4


@pytest.mark.parametrize("name", sorted(ROUTED_ALL))
def test_routed_and_dense_topk_both_match_the_oracle(name):
    """Token buckets (the default) and dense compute give the same translation."""
    wl = ROUTED_ALL[name]
    sk, sv, blob = inputs(wl, seed=13)
    tb, ts = _all_tokens(wl)
    ref = oracle.translate_tokens(wl, sk, sv, blob, tb, ts)
    ok = _clear_choice(wl, sk, sv, blob, tb, ts)
    tl = wl.translated_layers()
    assert ok[tl].mean() > 0.99
    outs = {}
    for routing in (1, 0):
        run = G.Run(wl, sk, sv, blob)
        assert M.mot_get_routing(run.h) == M.ROUTING_SPARSE
        M.mot_set_routing(run.h, routing)
        assert run.translate() == M.MOT_OK
        assert run.canaries_intact() and run.padding_untouched()
        got = run.gather(tb, ts)
        keep = np.broadcast_to(ok[..., None], got.shape)
        G.assert_parity(wl, got[tl][keep[tl]], ref[tl][keep[tl]], f"{name} routing {routing}")
        outs[routing] = got
    keep = np.broadcast_to(ok[..., None], outs[0].shape)
    diff = np.abs(outs[0] - outs[1])[tl][keep[tl]]
    assert diff.max() <= 2.0 ** -5   # fp32 summation order and one bf16 rounding apart


def test_expert_counts_match_the_oracle_choices():
    """mot_get_expert_counts: tokens per translator per group, as the fp64 gate
    chooses them (up to tokens at a near tie); usage statistics from them."""
    wl = TOPK_ROUTED["routed_top2_of4"]
    sk, sv, blob = inputs(wl, seed=14)
    run = G.Run(wl, sk, sv, blob)
    groups = 2 * len(wl.translated_layers())
    with pytest.raises(M.MotError) as e:   # nothing routed yet
        M.mot_get_expert_counts(run.h, groups, wl.n_translators)
    assert e.value.status == M.MOT_ERR_UNSUPPORTED
    assert run.translate() == M.MOT_OK
    counts = M.mot_get_expert_counts(run.h, groups, wl.n_translators)
    tb, ts = _all_tokens(wl)
    _, gate = oracle.translate_tokens(wl, sk, sv, blob, tb, ts, want_gate=True)
    ok = _clear_choice(wl, sk, sv, blob, tb, ts)
    n_tok = tb.size
    for r, l in enumerate(wl.translated_layers()):
        for x in (0, 1):
            g = 2 * r + x
            chosen = gate[l, x] > 0                       # [n][E]
            assert (chosen.sum(axis=1) == wl.top_k).all()
            ref = chosen.sum(axis=0)
            ties = int((~ok[l, x]).sum())
            assert counts[g].sum() == wl.top_k * n_tok
            assert np.abs(counts[g] - ref).max() <= ties, (g, counts[g], ref, ties)
    cv2, ent = M.expert_usage(counts)
    c = counts.astype(np.float64).ravel()
    assert cv2 == pytest.approx(c.var() / c.mean() ** 2)
    assert 0.0 < ent <= np.log(c.size) + 1e-12


def test_routing_switch_and_counter_errors():
    wl = SMALL["umma_ragged"]   # dense gate: no buckets to route
    sk, sv, blob = inputs(wl, seed=15)
    run = G.Run(wl, sk, sv, blob)
    assert M.mot_get_routing(run.h) == M.ROUTING_DENSE
    for bad, status in ((1, M.MOT_ERR_UNSUPPORTED), (2, M.MOT_ERR_INVALID_ARG),
                        (-1, M.MOT_ERR_INVALID_ARG)):
        with pytest.raises(M.MotError) as e:
            M.mot_set_routing(run.h, bad)
        assert e.value.status == status
    assert run.translate() == M.MOT_OK
    with pytest.raises(M.MotError) as e:
        M.mot_get_expert_counts(run.h, 2 * len(wl.translated_layers()), wl.n_translators)
    assert e.value.status == M.MOT_ERR_UNSUPPORTED
    wl2 = TOPK_ROUTED["routed_top1_of8"]
    sk2, sv2, blob2 = inputs(wl2, seed=15)
    run2 = G.Run(wl2, sk2, sv2, blob2)
    assert run2.translate() == M.MOT_OK
    with pytest.raises(M.MotError) as e:   # wrong element count
        M.mot_get_expert_counts(run2.h, 1, 3)
    assert e.value.status == M.MOT_ERR_INVALID_ARG


def test_routed_profile_and_launch_count():
    wl = TOPK_ROUTED["routed_top2_of4"]
    sk, sv, blob = inputs(wl, seed=16)
    run = G.Run(wl, sk, sv, blob)
    n0 = M.mot_get_launch_count(run.h)
    M.mot_profile_enable(run.h, True)
    assert run.translate() == M.MOT_OK
    stats = M.mot_profile_read(run.h)
    assert set(stats) == {"prep_tiles", "gate", "route_count", "route_plan", "route_fill", "pack",
                          "umma2_sparse_gemm1", "umma2_sparse_gemm2", "combine"}
    wl1 = TOPK_ROUTED["routed_top1_of8"]   # Top-1: GEMM2 stores the target rows, no combine
    sk1, sv1, blob1 = inputs(wl1, seed=16)
    run1 = G.Run(wl1, sk1, sv1, blob1)
    M.mot_profile_enable(run1.h, True)
    assert run1.translate() == M.MOT_OK
    assert "combine" not in M.mot_profile_read(run1.h)
    assert M.mot_get_launch_count(run.h) - n0 == sum(v[0] for v in stats.values())


# ---------------------------------------------------------------- failure detection

def test_bounded_wait_reports_timeout_and_the_context_survives():
    """A pipeline stage that is never filled makes a bounded wait run out: the
    kernels unwind, the status word reports MOT_ERR_TIMEOUT, and the next
    translation on the same context is correct."""
    wl = SMALL["umma_ragged"]
    sk, sv, blob = inputs(wl, seed=11)
    run = G.Run(wl, sk, sv, blob)
    M.mot_set_schedule(run.h, 0)
    M.mot_debug_set(run.h, True, 20_000_000)      # about 10 ms of SM cycles
    assert run.translate() == M.MOT_ERR_TIMEOUT
    assert M.mot_get_device_status(run.h) == M.MOT_OK   # reading cleared it
    M.mot_debug_set(run.h, False, 0)
    run.buf_k, run.dk = G.alloc_dst(wl)
    run.buf_v, run.dv = G.alloc_dst(wl)
    assert run.translate() == M.MOT_OK
    full_check(wl, run, sk, sv, blob, "after a timeout")


# ---------------------------------------------------------------- linearity in the gate

LIN = {
    "umma": synth.Workload("lin_umma", 3, 2, 64, 4, 2, 128, 3, 256, 3, 300, "bf16",
                           (300, 129, 1), layer_map=(2, -1, 0, 1)),
    "simt": synth.Workload("lin_simt", 2, 3, 16, 2, 5, 8, 3, 40, 2, 70, "bf16", (70, 33)),
}


def _fixed_gates(wl, seed):
    """Two gates on the simplex per (group, b, s) and their mixture at alpha = 0.3,
    fp32 [G][B][S][E]."""
    rng = np.random.default_rng(seed)
    G_ = 2 * len(wl.translated_layers())
    shape = (G_, wl.max_batch, wl.max_seq, wl.n_translators)
    g1 = rng.dirichlet(np.ones(wl.n_translators), size=shape[:3]).astype(np.float32)
    g2 = rng.dirichlet(np.ones(wl.n_translators) * 0.3, size=shape[:3]).astype(np.float32)
    alpha = 0.3
    g3 = (alpha * g1.astype(np.float64) + (1 - alpha) * g2.astype(np.float64)).astype(np.float32)
    return g1, g2, g3, alpha


def _oracle_gate(wl, g, tb, ts):
    """The [G][B][S][E] gate rows in the oracle's [L_t][2][n][E] layout."""
    out = np.zeros((wl.n_layers_tgt, 2, tb.size, wl.n_translators))
    for r, l in enumerate(wl.translated_layers()):
        for x in (0, 1):
            out[l, x] = g[2 * r + x][tb, ts]
    return out


@pytest.mark.parametrize("case,schedule", [("umma", 3), ("umma", 2), ("umma", 1), ("umma", 0),
                                           ("simt", 2)])
def test_fixed_gate_matches_oracle_and_combine_is_linear(case, schedule):
    """Eq. mot_definition on the GPU: with the gate rows given (test hook), the
    translation matches the oracle's with the same rows, and the translation of
    the mixed gate alpha g1 + (1 - alpha) g2 is alpha y(g1) + (1 - alpha) y(g2)
    within the outputs' rounding."""
    wl = LIN[case]
    sk, sv, blob = inputs(wl, seed=21)
    g1, g2, g3, alpha = _fixed_gates(wl, 5)
    tb = np.concatenate([np.full(L, b) for b, L in enumerate(wl.seq_lens)]).astype(np.int32)
    ts = np.concatenate([np.arange(L) for L in wl.seq_lens]).astype(np.int32)
    tl = wl.translated_layers()
    outs = []
    for g in (g1, g2, g3):
        run = G.Run(wl, sk, sv, blob)
        M.mot_set_schedule(run.h, schedule)
        gd = torch.from_numpy(g).cuda()
        M.mot_debug_fixed_gate(run.h, gd)
        assert run.translate() == M.MOT_OK
        M.mot_debug_fixed_gate(run.h, None)
        got = run.gather(tb, ts)[tl]
        ref = oracle.translate_tokens(wl, sk, sv, blob, tb, ts,
                                      gate_fixed=_oracle_gate(wl, g, tb, ts))[tl]
        G.assert_parity(wl, got, ref, f"{case} schedule {schedule} fixed gate")
        assert run.padding_untouched() and run.canaries_intact()
        outs.append(got)
    mix = alpha * outs[0] + (1 - alpha) * outs[1]
    G.assert_parity(wl, outs[2], mix, f"{case} schedule {schedule} linearity")
    # the hook is cleared: the next translation evaluates the gate again
    run = G.Run(wl, sk, sv, blob)
    assert run.translate() == M.MOT_OK
    ref = oracle.translate_tokens(wl, sk, sv, blob, tb, ts)[tl]
    G.assert_parity(wl, run.gather(tb, ts)[tl], ref, f"{case} evaluated gate")


# ---------------------------------------------------------------- outlier channels

OUTLIER = {
    "onchip": SMALL["umma_ragged"],
    "wide": synth.Workload("outlier_wide", 2, 12, 64, 2, 12, 64, 4, 1536, 2, 256, "bf16",
                           (256, 100)),
}


@pytest.mark.parametrize("case", sorted(OUTLIER))
def test_outlier_source_channels_stay_finite_and_within_the_bar(case):
    """Real K caches carry a few channels 10-100x the median scale. Scaling 4
    source channels of every layer by 100 enlarges the hidden pre-activations
    (rounded to fp16 on the tensor-core path) and the outputs (|y| up to ~100).
    The translation stays finite and within rel-RMS 1e-2; the max-abs bar of
    3e-2, set for outputs of unit scale, is scaled by the outputs' RMS (the
    fp16 rounding of the hidden values grows with them)."""
    wl = OUTLIER[case]
    sk, sv, blob = inputs(wl, seed=31)
    rng = np.random.default_rng(9)
    chans = rng.choice(wl.d_src, size=4, replace=False)
    for src in (sk, sv):
        f = H.storage_to_f64(wl, src)
        for c in chans:
            h, i = divmod(int(c), wl.src_head_dim)
            f[:, :, h, :, i] *= 100.0
        src[...] = H.to_storage(wl, f)
    run = G.Run(wl, sk, sv, blob)
    assert run.translate() == M.MOT_OK
    gk, gv = run.dst_f64()
    rk, rv = oracle.translate_full(wl, sk, sv, blob, run.seq[:run.batch])
    mask = G.translated_mask_full(wl, run.seq, run.batch)
    for got, ref, x in ((gk[mask], rk[mask], "K"), (gv[mask], rv[mask], "V")):
        assert np.isfinite(got).all()
        m = G.metrics(got, ref)
        rms = float(np.sqrt(np.mean(ref ** 2)))
        print(case, x, m, "rms(y)", rms)
        assert m["rel_rms"] <= 1e-2, (case, x, m)
        assert m["max_abs"] <= 3e-2 * max(1.0, rms), (case, x, m, rms)
