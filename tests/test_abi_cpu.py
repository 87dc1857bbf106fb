"""The C-ABI library without a GPU: it loads, exports every entry point that
include/mot.h declares, and rejects bad arguments before any CUDA call."""
import ctypes
import os
import re

import numpy as np

import pytest

from paper_2607_28979_gb300 import build as mot_build

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
mot_build.build()
import paper_2607_28979_gb300.mot as M   # noqa: E402


def declared_entry_points():
    text = open(os.path.join(ROOT, "include", "mot.h")).read()
    return sorted(set(re.findall(r"^(?:mot_status|const char\*)\s+(mot_\w+)\(", text, re.M)))


def test_every_declared_symbol_is_exported():
    names = declared_entry_points()
    assert len(names) >= 12
    for n in names:
        assert hasattr(M._lib, n), f"libmot.so does not export {n}"
    assert names == M.EXPORTED


def test_library_is_in_tree_and_has_no_cuda_runtime_dependency():
    assert os.path.dirname(M.LIB_PATH) == os.path.join(ROOT, "paper_2607_28979_gb300")


def test_status_strings():
    assert M.mot_status_string(M.MOT_OK) == "MOT_OK"
    assert M.mot_status_string(M.MOT_ERR_SEQ_LEN) == "MOT_ERR_SEQ_LEN"
    assert M.mot_status_string(M.MOT_ERR_TIMEOUT) == "MOT_ERR_TIMEOUT"
    assert M.mot_status_string(99) == "MOT_ERR_UNKNOWN"


GOOD = dict(n_layers_src=2, src_kv_heads=2, src_head_dim=64, n_layers_tgt=3, tgt_kv_heads=2,
            tgt_head_dim=128, n_translators=2, hidden=256, max_batch=2, max_seq=64)


@pytest.mark.parametrize("change,expect", [
    (dict(n_layers_src=0), M.MOT_ERR_INVALID_ARG),
    (dict(src_kv_heads=-1), M.MOT_ERR_INVALID_ARG),
    (dict(tgt_head_dim=0), M.MOT_ERR_INVALID_ARG),
    (dict(n_translators=0), M.MOT_ERR_INVALID_ARG),
    (dict(hidden=0), M.MOT_ERR_INVALID_ARG),
    (dict(max_batch=0), M.MOT_ERR_INVALID_ARG),
    (dict(max_seq=0), M.MOT_ERR_INVALID_ARG),
    (dict(top_k=3), M.MOT_ERR_INVALID_ARG),
    (dict(top_k=-1), M.MOT_ERR_INVALID_ARG),
    (dict(layer_map=[0, 2, 1]), M.MOT_ERR_INVALID_ARG),     # source layer 2 of 2
    (dict(layer_map=[0, -2, 1]), M.MOT_ERR_INVALID_ARG),
    (dict(n_translators=17, top_k=0), M.MOT_ERR_UNSUPPORTED),
    (dict(max_batch=4097), M.MOT_ERR_UNSUPPORTED),
])
def test_create_rejects_bad_config_before_cuda(change, expect):
    kw = dict(GOOD)
    kw.update(change)
    cfg = M.make_config(**kw)
    out = ctypes.c_void_p(123)
    assert M._lib.mot_create(ctypes.byref(cfg), ctypes.byref(out)) == expect
    assert out.value is None


def test_bad_dtype_rejected():
    cfg = M.make_config(**GOOD)
    cfg.dtype = 7
    out = ctypes.c_void_p()
    assert M._lib.mot_create(ctypes.byref(cfg), ctypes.byref(out)) == M.MOT_ERR_INVALID_ARG


def test_null_arguments():
    L = M._lib
    assert L.mot_create(None, None) == M.MOT_ERR_INVALID_ARG
    out = ctypes.c_void_p()
    assert L.mot_create(None, ctypes.byref(out)) == M.MOT_ERR_INVALID_ARG
    assert L.mot_load_weights(None, None, 0) == M.MOT_ERR_INVALID_ARG
    assert L.mot_translate(None, 16, 16, 16, 1, 16, 16, None) == M.MOT_ERR_INVALID_ARG
    assert L.mot_translate_host(None, 16, 16, 16, 1, 16, 16, None) == M.MOT_ERR_INVALID_ARG
    assert L.mot_get_device_status(None, None) == M.MOT_ERR_INVALID_ARG
    assert L.mot_destroy(None) == M.MOT_ERR_INVALID_ARG
    assert L.mot_get_path(None, None) == M.MOT_ERR_INVALID_ARG
    assert L.mot_profile_enable(None, 1) == M.MOT_ERR_INVALID_ARG
    assert L.mot_get_launch_count(None, None) == M.MOT_ERR_INVALID_ARG


def test_valid_config_without_gpu_is_a_cuda_error():
    torch = pytest.importorskip("torch")
    if torch.cuda.is_available():
        pytest.skip("a GPU is present")
    with pytest.raises(M.MotError) as e:
        M.mot_create(M.make_config(**GOOD))
    assert e.value.status == M.MOT_ERR_CUDA


def test_expert_usage_statistics_closed_forms():
    """CV^2 = Var(I) / Mean(I)^2 and entropy -sum p log p of p = I / sum I (Sec. 4.3),
    computed by the library's mot_expert_usage (host code, no GPU)."""
    import math
    cv2, ent = M.expert_usage([10, 10])          # balanced: no spread, log 2 nats
    assert cv2 == 0.0 and ent == pytest.approx(math.log(2), abs=1e-15)
    cv2, ent = M.expert_usage([20, 0])           # collapsed onto one translator
    assert cv2 == pytest.approx(1.0) and ent == 0.0
    cv2, ent = M.expert_usage([[6, 2], [1, 1]])  # counts of several groups pool
    c = [6, 2, 1, 1]
    mean = sum(c) / 4
    var = sum((x - mean) ** 2 for x in c) / 4
    assert cv2 == pytest.approx(var / mean ** 2)
    assert ent == pytest.approx(-sum(x / 10 * math.log(x / 10) for x in c))
    assert M.expert_usage([0, 0]) == (0.0, 0.0)
    with pytest.raises(M.MotError):
        M.expert_usage([3, -1])


def test_routing_calls_reject_null_handles():
    import numpy as np
    assert M._lib.mot_set_routing(None, 1) == M.MOT_ERR_INVALID_ARG
    v = ctypes.c_int32()
    assert M._lib.mot_get_routing(None, ctypes.byref(v)) == M.MOT_ERR_INVALID_ARG
    buf = np.zeros(4, dtype=np.int32)
    assert M._lib.mot_get_expert_counts(None, buf.ctypes.data, 4, None) == M.MOT_ERR_INVALID_ARG


RP_GOOD = dict(q_heads=12, kv_heads=2, head_dim=128, max_batch=4, max_seq=4096, top_s=128, n_full=2)


@pytest.mark.parametrize("change, expect", [
    (dict(q_heads=0), "MOT_ERR_INVALID_ARG"),
    (dict(kv_heads=0), "MOT_ERR_INVALID_ARG"),
    (dict(kv_heads=5), "MOT_ERR_INVALID_ARG"),      # 12 % 5: not a GQA grouping
    (dict(top_s=0), "MOT_ERR_INVALID_ARG"),
    (dict(n_full=-1), "MOT_ERR_INVALID_ARG"),
    (dict(max_seq=0), "MOT_ERR_INVALID_ARG"),
    (dict(head_dim=96), "MOT_ERR_UNSUPPORTED"),     # kernels take d in {64, 128}
    (dict(q_heads=20, kv_heads=2), "MOT_ERR_UNSUPPORTED"),   # group of 10: no instantiated kernel
])
def test_replay_create_rejects_bad_config_before_cuda(change, expect):
    kw = dict(RP_GOOD)
    kw.update(change)
    cfg = M.mot_replay_config(*[kw[k] for k in ("q_heads", "kv_heads", "head_dim", "max_batch",
                                                "max_seq", "top_s", "n_full")])
    out = ctypes.c_void_p(1)
    assert M._lib.mot_create_replay(ctypes.byref(cfg), ctypes.byref(out)) == getattr(M, expect)
    assert not out.value   # no handle on failure


def test_backbone_create_rejects_bad_window_before_cuda():
    import synth
    wl = synth.WORKLOADS["bt_gpt2s_opt125m"]
    cfg, bt = M.bt_config_from(wl)
    out = ctypes.c_void_p(1)
    for field, value in (("win_len", 0), ("win_start", -1), ("win_start", wl.n_layers_tgt),
                         ("heads", 0), ("heads", 5)):   # width 128 not a multiple of 5 heads
        bad = M.mot_bt_config(*[getattr(bt, f) for f, _ in M.mot_bt_config._fields_])
        setattr(bad, field, value)
        assert M._lib.mot_create_bt(ctypes.byref(cfg), ctypes.byref(bad),
                                    ctypes.byref(out)) == M.MOT_ERR_INVALID_ARG, field
        assert not out.value
    assert M._lib.mot_create_bt(None, ctypes.byref(bt), ctypes.byref(out)) == M.MOT_ERR_INVALID_ARG


def test_replay_backbone_and_debug_calls_reject_null_handles():
    L = M._lib
    assert L.mot_replay_attention(None, 0, None, None, None, None, None, 0, None, None) == M.MOT_ERR_INVALID_ARG
    assert L.mot_replay_select(None, None, None, 0, None, None) == M.MOT_ERR_INVALID_ARG
    assert L.mot_translate_bt(None, None, None, None, 0, None, None, None) == M.MOT_ERR_INVALID_ARG
    assert L.mot_debug_set(None, 0, 0) == M.MOT_ERR_INVALID_ARG
    assert L.mot_debug_fixed_gate(None, None) == M.MOT_ERR_INVALID_ARG
    assert L.mot_debug_gelu(3, None, None, 0, None, None) == M.MOT_ERR_INVALID_ARG
    assert L.mot_debug_gelu(0, None, None, -1, None, None) == M.MOT_ERR_INVALID_ARG
    assert L.mot_debug_gelu(0, None, None, 0, None, None) == M.MOT_OK   # nothing to do
    assert L.mot_debug_gelu(0, None, None, 4, None, None) == M.MOT_ERR_INVALID_ARG


def _static_call(cfg, weights, src_k, src_v, dst_k, dst_v, lens=0x9000, batch=1):
    """mot_translate_static with raw addresses (the checks below run before any
    CUDA call, so nothing is dereferenced)."""
    return M._lib.mot_translate_static(ctypes.byref(cfg), weights, src_k, src_v, lens, batch,
                                       dst_k, dst_v, None)


def test_static_entry_point_rejects_overlapping_outputs_before_cuda():
    import synth
    wl = synth.Workload("alias", 3, 2, 64, 4, 2, 128, 2, 256, 2, 64, "bf16", (64, 9))
    cfg = M.config_from(wl)
    sb = int(np.prod(wl.src_shape())) * 2
    db = int(np.prod(wl.dst_shape())) * 2
    wb = wl.blob_elems() * 2
    base = 1 << 40   # disjoint 16-byte-aligned address ranges
    w, sk, sv = base, base + (1 << 32), base + (2 << 32)
    dk, dv = base + (3 << 32), base + (4 << 32)
    # the same call without overlaps gets past these checks (no GPU: a CUDA error)
    ok = _static_call(cfg, w, sk, sv, dk, dv)
    assert ok != M.MOT_ERR_INVALID_ARG
    for args in ((w, sk, sv, sk, dv),                    # dst_k is src_k
                 (w, sk, sv, dk, sv),                    # dst_v is src_v
                 (w, sk, sv, sv + sb - 16, dv),          # dst_k runs into the tail of src_v
                 (w, sk, sv, dk, dk + db - 16),          # dst_v overlaps dst_k
                 (w, sk, sv, w + wb - 16, dv),           # dst_k over the weights' tail
                 (dv - wb + 16, sk, sv, dk, dv)):        # the weights' tail under dst_v
        assert _static_call(cfg, *args) == M.MOT_ERR_INVALID_ARG, args


def test_static_entry_point_rejects_huge_lengths_before_cuda():
    import synth
    wl = synth.Workload("huge", 2, 2, 64, 2, 2, 128, 2, 256, 1, 2**31 - 40, "bf16", (64,))
    cfg = M.config_from(wl)
    base = 1 << 44
    st = _static_call(cfg, base, base + (1 << 40), base + (2 << 40), base + (3 << 40),
                      base + (4 << 40))
    assert st == M.MOT_ERR_UNSUPPORTED
