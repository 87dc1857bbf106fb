"""The token-sampling bookkeeping of the full-size parity tests (no GPU)."""
import numpy as np

import oracle
import synth
import _helpers as H


def test_stratified_sample_covers_every_sequence_and_its_ends():
    lens = (32768, 16384, 8192, 4096)
    tb, ts = H.stratified_tokens(lens, 256, seed=1)
    assert 240 <= tb.size <= 300
    for b, L in enumerate(lens):
        s = ts[tb == b]
        assert 0 in s and L - 1 in s and (s < L).all() and np.unique(s).size == s.size
    # proportional to length
    assert (tb == 0).sum() > (tb == 3).sum()


def test_whole_tiles_are_aligned_windows_plus_the_last_tile():
    lens = (1024, 300, 0, 700)
    tb, ts = H.whole_tiles(lens, tile=256, seed=3)
    for b, L in enumerate(lens):
        s = ts[tb == b]
        if L == 0:
            assert s.size == 0
            continue
        assert (s < L).all()
    last = ts[tb == 3]
    assert 699 in last and 512 in last          # the final (ragged) window of the batch
    first = ts[tb == 0]
    assert first.size == 256 and first[0] % 256 == 0 and (np.diff(first) == 1).all()


def test_restricted_layers_reproduce_the_full_oracle():
    wl = synth.Workload("rl", 3, 2, 64, 4, 2, 128, 2, 256, 2, 300, "bf16", (300, 129))
    sk, sv, blob = synth.gen_cache(wl, 0), synth.gen_cache(wl, 1), synth.gen_weights(wl)
    lm = oracle.depth_ratio_map(3, 4)
    tb, ts = H.stratified_tokens(wl.seq_lens, 24)
    full = oracle.translate_tokens(wl, sk, sv, blob, tb, ts)
    wl2, b2 = H.restrict_layers(wl, blob, lm, {0, 3})
    part = oracle.translate_tokens(wl2, sk, sv, b2, tb, ts)
    np.testing.assert_array_equal(full[[0, 3]], part[[0, 3]])
    assert np.isnan(part[[1, 2]]).all()
