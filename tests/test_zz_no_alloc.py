"""mot_translate_static, the allocation-free entry point for callers that
cannot call cudaMalloc (for example a process whose device memory is divided
up front by its own pool allocator): its results must match the fp64 oracle
at the same bars as mot_translate, on two calls in a row (the second reuses
the shared scratch array the first left behind), and agree with mot_translate
within the bar. This file is collected last so that a run stopping at the
first failure has already run every other test."""
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

CASES = {
    "tiny_fp32": synth.WORKLOADS["tiny_fp32"],
    "bf16_ragged": synth.Workload("bf16_ragged", 3, 2, 64, 4, 2, 128, 2, 256, 4, 300, "bf16",
                                  (300, 129, 1), layer_map=(2, -1, 0, 1)),
    "bf16_topk": synth.Workload("bf16_topk", 2, 3, 16, 3, 5, 8, 4, 40, 2, 70, "bf16", (70, 33),
                                top_k=2),
}


@pytest.mark.parametrize("name", sorted(CASES))
def test_static_entry_point_matches_the_oracle_twice(name):
    wl = CASES[name]
    sk, sv, blob = (synth.gen_cache(wl, 0, 5), synth.gen_cache(wl, 1, 5),
                    synth.gen_weights(wl, 5))
    ref = G.Run(wl, sk, sv, blob)
    assert ref.translate() == M.MOT_OK
    lib_k, lib_v = ref.dst_f64()
    want_k, want_v = oracle.translate_full(wl, sk, sv, blob, ref.seq[:ref.batch])
    mask = G.translated_mask_full(wl, ref.seq, ref.batch)
    weights = G.to_device(wl, blob)
    cfg = M.config_from(wl)
    stream = torch.cuda.current_stream()
    for call in range(2):
        buf_k, dk = G.alloc_dst(wl)
        buf_v, dv = G.alloc_dst(wl)
        M.mot_translate_static(cfg, weights, ref.sk, ref.sv, ref.lens, ref.batch, dk, dv, stream)
        stream.synchronize()
        for got, want, lib, buf, x in ((dk, want_k, lib_k, buf_k, "K"),
                                       (dv, want_v, lib_v, buf_v, "V")):
            g = got.double().cpu().numpy()
            G.assert_parity(wl, g[mask], want[mask], f"{name} call {call} {x} vs oracle")
            # both paths sit within the bar of the oracle, so within twice the bar of each other
            m = G.metrics(g[mask], lib[mask])
            tol = G.TOL[wl.dtype]
            assert m["rel_rms"] <= 2 * tol["rel_rms"] and m["max_abs"] <= 2 * tol["max_abs"], \
                f"{name} call {call} {x} vs mot_translate: {m}"
            n = got.numel()
            s = G.sentinel_value(wl)
            assert bool((G.int_view(got)[torch.from_numpy(~mask).cuda()] == s).all()), \
                f"{name} call {call} {x}: wrote a position it must not touch"
            assert bool((G.int_view(buf[n:]) == s).all()), f"{name} call {call} {x}: past the end"


def test_static_entry_point_rejects_oversized_problems():
    wl = synth.WORKLOADS["gpt2s_opt125m"]   # needs 8 * 1024 * 4 * 1540 * 4 bytes > 64 MiB
    cfg = M.config_from(wl)
    lens = torch.tensor(wl.seq_lens, dtype=torch.int32, device="cuda")
    big = torch.empty(16, dtype=torch.int16, device="cuda")
    with pytest.raises(M.MotError) as e:
        M.mot_translate_static(cfg, big, big, big, lens, wl.batch, big, big)
    assert e.value.status == M.MOT_ERR_UNSUPPORTED
