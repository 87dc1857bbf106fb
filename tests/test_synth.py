"""The seeded generator: published SplitMix64 outputs, distribution and layout."""
import numpy as np

import synth


def test_splitmix64_reference_outputs():
    # SplitMix64 started from state 0: the first outputs of the published generator.
    assert [synth.splitmix64(0, n) for n in range(3)] == [
        0xE220A8397B1DCDAF, 0x6E789E6AA1B965F4, 0x06C45D188009454F]


def test_normal_draws_are_standard_and_reproducible():
    a = synth.normal(0, 7, 400_000)
    assert abs(a.mean()) < 5e-3 and abs(a.std() - 1.0) < 5e-3
    assert np.array_equal(a, synth.normal(0, 7, 400_000))
    assert not np.array_equal(a[:100], synth.normal(1, 7, 100))
    assert not np.array_equal(a[:100], synth.normal(0, 8, 100))


def test_cache_and_blob_layout():
    wl = synth.WORKLOADS["tiny_fp32"].replace(n_layers_src=2, n_layers_tgt=2, hidden=64,
                                              src_kv_heads=2, tgt_kv_heads=2)
    k = synth.gen_cache(wl, 0)
    v = synth.gen_cache(wl, 1)
    assert k.shape == wl.src_shape() and k.dtype == np.float32
    assert not np.array_equal(k, v)
    # per-channel scale: the spread of channel std devs is lognormal-like (not all 1)
    ch_std = k[0, 0].transpose(0, 2, 1).reshape(-1, wl.max_seq).std(axis=1)
    assert ch_std.min() < 0.7 and ch_std.max() > 1.4
    blob = synth.gen_weights(wl)
    assert blob.size == wl.blob_elems()
    offs = list(synth.blob_offsets(wl))
    l, x, t, m, off, n, fan_in = offs[2]          # first W1 block
    assert t == synth.T_W1 and fan_in == wl.d_src
    w1 = blob[off:off + n].astype(np.float64)
    assert abs(w1.std() * np.sqrt(fan_in) - 1.0) < 0.02


def test_bf16_rounding():
    wl = synth.WORKLOADS["gpt2s_opt125m"].replace(n_layers_src=1, max_batch=1, max_seq=8,
                                                  seq_lens=(8,))
    k = synth.gen_cache(wl, 0)
    assert k.dtype == np.uint16
    f = (k.astype(np.uint32) << 16).view(np.float32)
    assert np.isfinite(f).all() and 0.5 < f.std() < 3.0
