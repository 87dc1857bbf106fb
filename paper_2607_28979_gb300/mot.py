"""Python binding of ``libmot.so``: argument marshalling only.

Every step of the translation runs in the CUDA library (``csrc/``). This
module loads it with ctypes and exposes its C entry points under the same
names. There is no CPU fallback: if the library is missing, importing this
package raises ``ImportError`` (build it with ``python -m
paper_2607_28979_gb300.build`` or ``__graft_entry__.build()``).

Tensor arguments may be ``torch.Tensor`` objects (their ``data_ptr()`` is
passed) or plain integers holding device / host addresses. Streams may be a
``torch.cuda.Stream``, an integer handle, or ``None`` (the current torch
stream if torch is loaded, else the legacy default stream).
"""
from __future__ import annotations

import ctypes
import os
import sys
from typing import Optional, Sequence

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "libmot.so")

if not os.path.exists(LIB_PATH):
    raise ImportError(f"libmot.so is not built ({LIB_PATH}); run "
                      "`python -m paper_2607_28979_gb300.build` first")

_lib = ctypes.CDLL(LIB_PATH)

# ---------------------------------------------------------------- C types

MOT_OK, MOT_ERR_INVALID_ARG, MOT_ERR_UNSUPPORTED, MOT_ERR_NO_WEIGHTS, MOT_ERR_WEIGHTS_SIZE, \
    MOT_ERR_OOM, MOT_ERR_CUDA, MOT_ERR_SEQ_LEN, MOT_ERR_TIMEOUT = range(9)
MOT_BF16, MOT_FP32 = 0, 1


class mot_config(ctypes.Structure):
    _fields_ = [("n_layers_src", ctypes.c_int32), ("src_kv_heads", ctypes.c_int32),
                ("src_head_dim", ctypes.c_int32), ("n_layers_tgt", ctypes.c_int32),
                ("tgt_kv_heads", ctypes.c_int32), ("tgt_head_dim", ctypes.c_int32),
                ("n_translators", ctypes.c_int32), ("top_k", ctypes.c_int32),
                ("hidden", ctypes.c_int32), ("max_batch", ctypes.c_int32),
                ("max_seq", ctypes.c_int32), ("dtype", ctypes.c_int32),
                ("layer_map", ctypes.POINTER(ctypes.c_int32))]


class mot_h_config(ctypes.Structure):
    _fields_ = [("n_layers_src", ctypes.c_int32), ("src_act_dim", ctypes.c_int32),
                ("n_layers_tgt", ctypes.c_int32), ("tgt_act_dim", ctypes.c_int32),
                ("tgt_kv_heads", ctypes.c_int32), ("tgt_head_dim", ctypes.c_int32),
                ("n_translators", ctypes.c_int32), ("top_k", ctypes.c_int32),
                ("hidden", ctypes.c_int32), ("max_batch", ctypes.c_int32),
                ("max_seq", ctypes.c_int32), ("dtype", ctypes.c_int32),
                ("layer_map", ctypes.POINTER(ctypes.c_int32))]


class mot_bt_config(ctypes.Structure):
    _fields_ = [("win_start", ctypes.c_int32), ("win_len", ctypes.c_int32),
                ("width", ctypes.c_int32), ("heads", ctypes.c_int32), ("ffn", ctypes.c_int32)]


class mot_replay_config(ctypes.Structure):
    _fields_ = [("q_heads", ctypes.c_int32), ("kv_heads", ctypes.c_int32),
                ("head_dim", ctypes.c_int32), ("max_batch", ctypes.c_int32),
                ("max_seq", ctypes.c_int32), ("top_s", ctypes.c_int32), ("n_full", ctypes.c_int32)]


class mot_kernel_stat(ctypes.Structure):
    _fields_ = [("name", ctypes.c_char * 32), ("launches", ctypes.c_int64),
                ("total_ms", ctypes.c_double)]


_H = ctypes.c_void_p
_P = ctypes.c_void_p
_S = ctypes.c_int

_SIGS = {
    "mot_create": [ctypes.POINTER(mot_config), ctypes.POINTER(ctypes.c_void_p)],
    "mot_load_weights": [_H, _P, ctypes.c_size_t],
    "mot_translate": [_H, _P, _P, _P, ctypes.c_int32, _P, _P, _P],
    "mot_translate_host": [_H, _P, _P, _P, ctypes.c_int32, _P, _P, _P],
    "mot_get_device_status": [_H, _P],
    "mot_destroy": [_H],
    "mot_get_layer_map": [_H, _P, ctypes.c_int32],
    "mot_get_path": [_H, ctypes.POINTER(ctypes.c_int32)],
    "mot_set_schedule": [_H, ctypes.c_int32],
    "mot_get_schedule": [_H, ctypes.POINTER(ctypes.c_int32)],
    "mot_profile_enable": [_H, ctypes.c_int32],
    "mot_profile_read": [_H, ctypes.POINTER(mot_kernel_stat), ctypes.c_int32,
                         ctypes.POINTER(ctypes.c_int32)],
    "mot_get_launch_count": [_H, ctypes.POINTER(ctypes.c_int64)],
    "mot_create_h": [ctypes.POINTER(mot_h_config), ctypes.POINTER(ctypes.c_void_p)],
    "mot_translate_h": [_H, _P, _P, ctypes.c_int32, _P, _P, _P],
    "mot_set_routing": [_H, ctypes.c_int32],
    "mot_get_routing": [_H, ctypes.POINTER(ctypes.c_int32)],
    "mot_get_expert_counts": [_H, _P, ctypes.c_int32, _P],
    "mot_expert_usage": [_P, ctypes.c_int32, _P, _P],
    "mot_debug_set": [_H, ctypes.c_int32, ctypes.c_int64],
    "mot_debug_gelu": [ctypes.c_int32, _P, _P, ctypes.c_int64, _P, _P],
    "mot_debug_fixed_gate": [_H, _P],
    "mot_translate_static": [ctypes.POINTER(mot_config), _P, _P, _P, _P, ctypes.c_int32, _P, _P,
                             _P],
    "mot_create_bt": [ctypes.POINTER(mot_config), ctypes.POINTER(mot_bt_config),
                      ctypes.POINTER(ctypes.c_void_p)],
    "mot_translate_bt": [_H, _P, _P, _P, ctypes.c_int32, _P, _P, _P],
    "mot_create_replay": [ctypes.POINTER(mot_replay_config), ctypes.POINTER(ctypes.c_void_p)],
    "mot_replay_attention": [_H, ctypes.c_int32, _P, _P, _P, _P, _P, ctypes.c_int32, _P, _P],
    "mot_replay_select": [_H, _P, _P, ctypes.c_int32, _P, _P],
}
for _name, _args in _SIGS.items():
    _f = getattr(_lib, _name)
    _f.argtypes = _args
    _f.restype = _S
_lib.mot_status_string.argtypes = [_S]
_lib.mot_status_string.restype = ctypes.c_char_p

# Names declared by include/mot.h, for the export check.
EXPORTED = sorted(list(_SIGS) + ["mot_status_string"])


class MotError(RuntimeError):
    def __init__(self, status: int, where: str):
        self.status = status
        super().__init__(f"{where}: {mot_status_string(status)}")


def mot_status_string(status: int) -> str:
    return _lib.mot_status_string(int(status)).decode()


def _check(status: int, where: str) -> None:
    if status != MOT_OK:
        raise MotError(status, where)


def _addr(x) -> Optional[int]:
    if x is None:
        return None
    if isinstance(x, int):
        return x
    if hasattr(x, "data_ptr"):
        return x.data_ptr()
    if hasattr(x, "ctypes"):   # numpy array (host buffers)
        return x.ctypes.data
    raise TypeError(f"cannot take the address of {type(x)}")


def _stream(s) -> Optional[int]:
    if s is None:
        torch = sys.modules.get("torch")
        if torch is not None and torch.cuda.is_available() and torch.cuda.is_initialized():
            return torch.cuda.current_stream().cuda_stream
        return None
    if isinstance(s, int):
        return s
    return s.cuda_stream


# ---------------------------------------------------------------- entry points

class Handle:
    """Owns one ``mot_handle``; destroyed with ``mot_destroy`` or on GC."""

    def __init__(self, ptr: int, n_layers_tgt: int):
        self.ptr = ptr
        self.n_layers_tgt = n_layers_tgt

    def __del__(self):
        if getattr(self, "ptr", None):
            try:
                _lib.mot_destroy(self.ptr)
            except Exception:
                pass
            self.ptr = None


def make_config(n_layers_src, src_kv_heads, src_head_dim, n_layers_tgt, tgt_kv_heads,
                tgt_head_dim, n_translators, hidden, max_batch, max_seq, dtype="bf16", top_k=0,
                layer_map: Optional[Sequence[int]] = None):
    cfg = mot_config(n_layers_src, src_kv_heads, src_head_dim, n_layers_tgt, tgt_kv_heads,
                     tgt_head_dim, n_translators, top_k, hidden, max_batch, max_seq,
                     MOT_BF16 if dtype in ("bf16", MOT_BF16) else MOT_FP32, None)
    keep = None
    if layer_map is not None:
        keep = (ctypes.c_int32 * len(layer_map))(*layer_map)
        cfg.layer_map = ctypes.cast(keep, ctypes.POINTER(ctypes.c_int32))
    cfg._keep = keep   # keep the array alive as long as the struct
    return cfg


def config_from(wl):
    """mot_config for any object with the Workload field names."""
    return make_config(wl.n_layers_src, wl.src_kv_heads, wl.src_head_dim, wl.n_layers_tgt,
                       wl.tgt_kv_heads, wl.tgt_head_dim, wl.n_translators, wl.hidden,
                       wl.max_batch, wl.max_seq, wl.dtype, wl.top_k, wl.layer_map)


def h_config_from(wl):
    """mot_h_config (MoT-h) for a Workload with ``act_tgt`` > 0 (the source
    activation stored as a one-head cache of width ``src_head_dim``)."""
    cfg = mot_h_config(wl.n_layers_src, wl.src_head_dim, wl.n_layers_tgt, wl.act_tgt,
                       wl.tgt_kv_heads, wl.tgt_head_dim, wl.n_translators, wl.top_k, wl.hidden,
                       wl.max_batch, wl.max_seq, MOT_BF16 if wl.dtype == "bf16" else MOT_FP32)
    if wl.layer_map is not None:
        arr = (ctypes.c_int32 * len(wl.layer_map))(*wl.layer_map)
        cfg.layer_map = ctypes.cast(arr, ctypes.POINTER(ctypes.c_int32))
        cfg._keep = arr
    return cfg


def mot_create_h(cfg: mot_h_config) -> Handle:
    out = ctypes.c_void_p()
    _check(_lib.mot_create_h(ctypes.byref(cfg), ctypes.byref(out)), "mot_create_h")
    return Handle(out.value, cfg.n_layers_tgt)


def mot_translate_h(h: Handle, src_act, seq_lens, batch: int, dst_k, dst_v, stream=None) -> None:
    _check(_lib.mot_translate_h(h.ptr, _addr(src_act), _addr(seq_lens), int(batch), _addr(dst_k),
                                _addr(dst_v), _stream(stream)), "mot_translate_h")


def bt_config_from(wl):
    """(mot_config, mot_bt_config) for a Workload with backbone translators (``bt``)."""
    return config_from(wl), mot_bt_config(*wl.bt)


def mot_create_bt(cfg: mot_config, bt: mot_bt_config) -> Handle:
    out = ctypes.c_void_p()
    _check(_lib.mot_create_bt(ctypes.byref(cfg), ctypes.byref(bt), ctypes.byref(out)),
           "mot_create_bt")
    return Handle(out.value, cfg.n_layers_tgt)


def mot_translate_bt(h: Handle, src_k, src_v, seq_lens, batch: int, dst_k, dst_v,
                     stream=None) -> None:
    _check(_lib.mot_translate_bt(h.ptr, _addr(src_k), _addr(src_v), _addr(seq_lens), int(batch),
                                 _addr(dst_k), _addr(dst_v), _stream(stream)), "mot_translate_bt")


def replay_config_from(wl):
    """mot_replay_config for a ``synth.ReplayWorkload``."""
    return mot_replay_config(wl.q_heads, wl.kv_heads, wl.head_dim, wl.max_batch, wl.max_seq,
                             wl.top_s, wl.n_full)


def mot_create_replay(cfg: mot_replay_config) -> Handle:
    out = ctypes.c_void_p()
    _check(_lib.mot_create_replay(ctypes.byref(cfg), ctypes.byref(out)), "mot_create_replay")
    return Handle(out.value, 0)


def mot_replay_attention(h: Handle, layer: int, q, k, v, guide, seq_lens, batch: int, out,
                         stream=None) -> None:
    _check(_lib.mot_replay_attention(h.ptr, int(layer), _addr(q), _addr(k), _addr(v),
                                     _addr(guide), _addr(seq_lens), int(batch), _addr(out),
                                     _stream(stream)), "mot_replay_attention")


def mot_replay_select(h: Handle, guide, seq_lens, batch: int, sel, stream=None) -> None:
    _check(_lib.mot_replay_select(h.ptr, _addr(guide), _addr(seq_lens), int(batch), _addr(sel),
                                  _stream(stream)), "mot_replay_select")


def mot_create(cfg: mot_config) -> Handle:
    out = ctypes.c_void_p()
    _check(_lib.mot_create(ctypes.byref(cfg), ctypes.byref(out)), "mot_create")
    return Handle(out.value, cfg.n_layers_tgt)


def mot_load_weights(h: Handle, blob) -> None:
    """``blob``: host numpy array / bytes-like holding the packed weights."""
    if hasattr(blob, "ctypes"):
        ptr, nbytes = blob.ctypes.data, blob.nbytes
    else:
        buf = (ctypes.c_char * len(blob)).from_buffer_copy(blob)
        ptr, nbytes = ctypes.addressof(buf), len(blob)
    _check(_lib.mot_load_weights(h.ptr, ptr, nbytes), "mot_load_weights")


def mot_translate(h: Handle, src_k, src_v, seq_lens, batch: int, dst_k, dst_v, stream=None) -> None:
    _check(_lib.mot_translate(h.ptr, _addr(src_k), _addr(src_v), _addr(seq_lens), int(batch),
                              _addr(dst_k), _addr(dst_v), _stream(stream)), "mot_translate")


def mot_translate_host(h: Handle, src_k, src_v, seq_lens, batch: int, dst_k, dst_v,
                       stream=None) -> None:
    _check(_lib.mot_translate_host(h.ptr, _addr(src_k), _addr(src_v), _addr(seq_lens), int(batch),
                                   _addr(dst_k), _addr(dst_v), _stream(stream)),
           "mot_translate_host")


MOT_STATIC_SCRATCH_BYTES = 64 << 20


def mot_translate_static(cfg: mot_config, weights, src_k, src_v, seq_lens, batch: int, dst_k,
                         dst_v, stream=None) -> None:
    """Allocation-free translation: no handle, weights (packed blob) in device memory."""
    _check(_lib.mot_translate_static(ctypes.byref(cfg), _addr(weights), _addr(src_k),
                                     _addr(src_v), _addr(seq_lens), int(batch), _addr(dst_k),
                                     _addr(dst_v), _stream(stream)), "mot_translate_static")


def mot_debug_fixed_gate(h: Handle, gate) -> None:
    """Use the gate rows in `gate` (device float [G][max_batch][max_seq][E]) until
    cleared with None."""
    _check(_lib.mot_debug_fixed_gate(h.ptr, _addr(gate)), "mot_debug_fixed_gate")


GELU_FORM_MLP, GELU_FORM_BACKBONE, GELU_FORM_SIMT = 0, 1, 2


def mot_debug_gelu(form: int, u, gate, out, stream=None) -> None:
    """out = GELU(u) * gate with the device GELU form `form` (float32 device tensors)."""
    _check(_lib.mot_debug_gelu(int(form), _addr(u), _addr(gate), int(u.numel()), _addr(out),
                               _stream(stream)), "mot_debug_gelu")


def mot_get_device_status(h: Handle, stream=None) -> int:
    """Returns the status code (does not raise for device-reported errors)."""
    return _lib.mot_get_device_status(h.ptr, _stream(stream))


def mot_destroy(h: Handle) -> None:
    if h.ptr:
        ptr, h.ptr = h.ptr, None
        _check(_lib.mot_destroy(ptr), "mot_destroy")


def mot_get_layer_map(h: Handle) -> list:
    arr = (ctypes.c_int32 * h.n_layers_tgt)()
    _check(_lib.mot_get_layer_map(h.ptr, arr, h.n_layers_tgt), "mot_get_layer_map")
    return list(arr)


def mot_get_path(h: Handle) -> int:
    p = ctypes.c_int32()
    _check(_lib.mot_get_path(h.ptr, ctypes.byref(p)), "mot_get_path")
    return p.value


SCHEDULE_SPLIT, SCHEDULE_FUSED, SCHEDULE_PAIR, SCHEDULE_ONCHIP = 0, 1, 2, 3


def mot_set_schedule(h: Handle, schedule: int) -> None:
    _check(_lib.mot_set_schedule(h.ptr, int(schedule)), "mot_set_schedule")


def mot_get_schedule(h: Handle) -> int:
    v = ctypes.c_int32()
    _check(_lib.mot_get_schedule(h.ptr, ctypes.byref(v)), "mot_get_schedule")
    return v.value


def mot_debug_set(h: Handle, stall_test: bool, wait_limit_cycles: int = 0) -> None:
    _check(_lib.mot_debug_set(h.ptr, int(bool(stall_test)), int(wait_limit_cycles)), "mot_debug_set")


def mot_profile_enable(h: Handle, enable: bool = True) -> None:
    _check(_lib.mot_profile_enable(h.ptr, int(bool(enable))), "mot_profile_enable")


def mot_profile_read(h: Handle) -> dict:
    """{kernel name: (launches, total_ms)} since the last read."""
    cap = 16
    arr = (mot_kernel_stat * cap)()
    n = ctypes.c_int32()
    _check(_lib.mot_profile_read(h.ptr, arr, cap, ctypes.byref(n)), "mot_profile_read")
    return {arr[i].name.decode(): (arr[i].launches, arr[i].total_ms) for i in range(n.value)}


def mot_get_launch_count(h: Handle) -> int:
    c = ctypes.c_int64()
    _check(_lib.mot_get_launch_count(h.ptr, ctypes.byref(c)), "mot_get_launch_count")
    return c.value


ROUTING_DENSE, ROUTING_SPARSE = 0, 1


def mot_set_routing(h: Handle, routing: int) -> None:
    _check(_lib.mot_set_routing(h.ptr, int(routing)), "mot_set_routing")


def mot_get_routing(h: Handle) -> int:
    v = ctypes.c_int32()
    _check(_lib.mot_get_routing(h.ptr, ctypes.byref(v)), "mot_get_routing")
    return v.value


def mot_get_expert_counts(h: Handle, n_groups: int, n_translators: int, stream=None):
    """Tokens routed to each translator of each (layer, K/V) group by the last
    translation: an int32 array [n_groups][n_translators]."""
    import numpy as np
    out = np.zeros((n_groups, n_translators), dtype=np.int32)
    _check(_lib.mot_get_expert_counts(h.ptr, out.ctypes.data, out.size, _stream(stream)),
           "mot_get_expert_counts")
    return out


def expert_usage(counts):
    """Translator usage statistics over selection counts I_e (Sec. 4.3), all
    groups pooled: (Var(I) / Mean(I)^2, -sum p_e ln p_e). Computed by the
    library's mot_expert_usage."""
    import numpy as np
    c = np.ascontiguousarray(np.asarray(counts).ravel(), dtype=np.int32)
    cv2, ent = ctypes.c_double(), ctypes.c_double()
    _check(_lib.mot_expert_usage(c.ctypes.data, int(c.size), ctypes.byref(cv2), ctypes.byref(ent)),
           "mot_expert_usage")
    return cv2.value, ent.value
