"""fp64 CPU oracle for the MoT KV-cache translation pass (ctypes wrapper).

TEST INFRASTRUCTURE. Only the tests, ``__graft_entry__.smoke()`` and the
CPU-baseline / reference legs of ``bench.py`` may import this package. The
product path (the ``paper_2607_28979_gb300`` package and its CUDA library)
never imports, links or runs it, and this package imports nothing from there.

The arithmetic lives in ``mot_oracle.c``; its header states what is computed
(Def. 3.1 / Eq. mot_definition, the App. C.2 translator read as the configs'
Linear-GELU-Linear MLP, the App. C.3 depth-ratio map) and how each part is pinned.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
from typing import Optional, Sequence

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "mot_oracle.c")
_SRCS = (_SRC, os.path.join(_HERE, "bt_oracle.c"), os.path.join(_HERE, "replay_oracle.c"))
_LIB = os.path.join(_HERE, "libmot_oracle.so")


class OracleDims(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int32) for n in
                ("L_s", "H_s", "d_s", "L_t", "H_t", "d_t", "E", "top_k", "H", "B", "S", "dtype")]


class OracleReplayDims(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int32) for n in ("B", "N", "Hq", "Hkv", "d", "S", "n_full")]


class OracleBtDims(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int32) for n in ("win_start", "win_len", "width", "heads", "ffn")]


def build(force: bool = False) -> str:
    """Compile ``libmot_oracle.so`` next to its source if missing or stale."""
    stale = not os.path.exists(_LIB) or any(os.path.getmtime(_LIB) < os.path.getmtime(f)
                                             for f in _SRCS)
    if force or stale:
        tmp = _LIB + f".{os.getpid()}.tmp"
        subprocess.check_call(["gcc", "-O2", "-fopenmp", "-shared", "-fPIC", "-o", tmp, *_SRCS,
                               "-lm"])
        os.replace(tmp, _LIB)
    return _LIB


_lib = None


def _load():
    global _lib
    if _lib is None:
        lib = ctypes.CDLL(build())
        P = ctypes.c_void_p
        lib.oracle_depth_ratio_map.restype = ctypes.c_int
        lib.oracle_depth_ratio_map.argtypes = [ctypes.c_int32, ctypes.c_int32, P]
        lib.oracle_gelu.restype = ctypes.c_double
        lib.oracle_gelu.argtypes = [ctypes.c_double]
        lib.oracle_bf16_to_double.restype = ctypes.c_double
        lib.oracle_bf16_to_double.argtypes = [ctypes.c_uint16]
        lib.oracle_gate_from_logits.restype = None
        lib.oracle_gate_from_logits.argtypes = [P, ctypes.c_int, ctypes.c_int, P]
        lib.oracle_translate_tokens.restype = ctypes.c_int
        lib.oracle_translate_tokens.argtypes = [ctypes.POINTER(OracleDims), P, P, P, P,
                                                ctypes.c_int64, P, P, P, P, P]
        lib.oracle_translate_h_tokens.restype = ctypes.c_int
        lib.oracle_translate_h_tokens.argtypes = [ctypes.POINTER(OracleDims), ctypes.c_int32, P,
                                                  P, P, ctypes.c_int64, P, P, P, P, P]
        lib.oracle_translate_full.restype = ctypes.c_int
        lib.oracle_translate_full.argtypes = [ctypes.POINTER(OracleDims), P, P, P, P,
                                              ctypes.c_int32, P, P, P]
        lib.oracle_layernorm.restype = None
        lib.oracle_layernorm.argtypes = [P, ctypes.c_int64, P, P, P]
        lib.oracle_bt_attention.restype = ctypes.c_int
        lib.oracle_bt_attention.argtypes = [ctypes.c_int, ctypes.c_int, ctypes.c_int, P, P, P, P]
        lib.oracle_bt_blob_elems.restype = ctypes.c_int64
        lib.oracle_bt_blob_elems.argtypes = [ctypes.POINTER(OracleDims),
                                             ctypes.POINTER(OracleBtDims)]
        lib.oracle_bt_backbone.restype = ctypes.c_int
        lib.oracle_bt_backbone.argtypes = [ctypes.POINTER(OracleDims), ctypes.POINTER(OracleBtDims),
                                           P, ctypes.c_int, ctypes.c_int, P, P, P]
        lib.oracle_bt_tokens.restype = ctypes.c_int
        lib.oracle_bt_tokens.argtypes = [ctypes.POINTER(OracleDims), ctypes.POINTER(OracleBtDims),
                                         P, P, P, P, ctypes.c_int64, P, P, P, P, P]
        RD = ctypes.POINTER(OracleReplayDims)
        lib.oracle_replay_select.restype = ctypes.c_int
        lib.oracle_replay_select.argtypes = [RD, P, ctypes.c_int, ctypes.c_int, P]
        lib.oracle_replay_query.restype = ctypes.c_int
        lib.oracle_replay_query.argtypes = [RD, ctypes.c_int, P, P, P, P, ctypes.c_int,
                                            ctypes.c_int, ctypes.c_int, P]
        lib.oracle_replay_tokens.restype = ctypes.c_int
        lib.oracle_replay_tokens.argtypes = [RD, ctypes.c_int, P, P, P, P, ctypes.c_int64, P, P,
                                             P, P]
        _lib = lib
    return _lib


def _ptr(a: Optional[np.ndarray]):
    return None if a is None else a.ctypes.data


def dims_of(wl) -> OracleDims:
    """OracleDims for a ``synth.Workload``-like object."""
    return OracleDims(wl.n_layers_src, wl.src_kv_heads, wl.src_head_dim,
                      wl.n_layers_tgt, wl.tgt_kv_heads, wl.tgt_head_dim,
                      wl.n_translators, wl.top_k, wl.hidden, wl.max_batch, wl.max_seq,
                      0 if wl.dtype == "bf16" else 1)


def depth_ratio_map(L_s: int, L_t: int) -> list:
    out = np.zeros(L_t, dtype=np.int32)
    if _load().oracle_depth_ratio_map(L_s, L_t, out.ctypes.data) != 0:
        raise ValueError("invalid layer counts")
    return out.tolist()


def gelu(x: float) -> float:
    return float(_load().oracle_gelu(float(x)))


def bf16_to_double(bits: int) -> float:
    return float(_load().oracle_bf16_to_double(bits))


def gate_from_logits(logits: Sequence[float], top_k: int = 0) -> np.ndarray:
    lg = np.ascontiguousarray(logits, dtype=np.float64)
    g = np.empty_like(lg)
    _load().oracle_gate_from_logits(lg.ctypes.data, lg.size, top_k, g.ctypes.data)
    return g


def _map_arr(layer_map):
    return None if layer_map is None else np.ascontiguousarray(layer_map, dtype=np.int32)


def translate_tokens(wl, src_k, src_v, blob, tok_b, tok_s, gate_fixed=None, want_gate=False):
    """Translate sampled tokens. Returns out[L_t][2][n][D_t] (NaN for untranslated
    layers) and, if ``want_gate``, the kept renormalised gate [L_t][2][n][E]."""
    tb = np.ascontiguousarray(tok_b, dtype=np.int32)
    ts = np.ascontiguousarray(tok_s, dtype=np.int32)
    n = tb.size
    out = np.full((wl.n_layers_tgt, 2, n, wl.d_tgt), np.nan, dtype=np.float64)
    gate = np.full((wl.n_layers_tgt, 2, n, wl.n_translators), np.nan) if want_gate else None
    gf = None if gate_fixed is None else np.ascontiguousarray(gate_fixed, dtype=np.float64)
    lm = _map_arr(wl.layer_map)
    d = dims_of(wl)
    # bound to names: the C call must not see the address of a freed temporary copy
    k_c, v_c, w_c = (np.ascontiguousarray(a) for a in (src_k, src_v, blob))
    rc = _load().oracle_translate_tokens(ctypes.byref(d), _ptr(lm), _ptr(k_c), _ptr(v_c),
                                         _ptr(w_c), n, _ptr(tb), _ptr(ts),
                                         _ptr(gf), _ptr(out), _ptr(gate))
    if rc != 0:
        raise ValueError("oracle_translate_tokens: invalid arguments")
    return (out, gate) if want_gate else out


def translate_h_tokens(wl, src_act, blob, tok_b, tok_s, want_act=False):
    """MoT-h (App. C.5) for sampled tokens: the translated activation restored
    through the target's projections. Returns (K, V), each [L_t][n][D_t] (NaN
    for untranslated layers), and with ``want_act`` the activation [L_t][n][d_at]."""
    assert wl.is_h and wl.src_kv_heads == 1
    tb = np.ascontiguousarray(tok_b, dtype=np.int32)
    ts = np.ascontiguousarray(tok_s, dtype=np.int32)
    n = tb.size
    ok = np.full((wl.n_layers_tgt, n, wl.d_tgt), np.nan, dtype=np.float64)
    ov = np.full_like(ok, np.nan)
    act = np.full((wl.n_layers_tgt, n, wl.act_tgt), np.nan) if want_act else None
    lm = _map_arr(wl.layer_map)
    a_c, w_c = np.ascontiguousarray(src_act), np.ascontiguousarray(blob)
    rc = _load().oracle_translate_h_tokens(ctypes.byref(dims_of(wl)), wl.act_tgt, _ptr(lm),
                                           _ptr(a_c), _ptr(w_c), n, _ptr(tb), _ptr(ts),
                                           _ptr(ok), _ptr(ov), _ptr(act))
    if rc != 0:
        raise ValueError("oracle_translate_h_tokens: invalid arguments")
    return (ok, ov, act) if want_act else (ok, ov)


def translate_full(wl, src_k, src_v, blob, seq_lens, fill=np.nan):
    """Full translation into double caches shaped like the target cache."""
    sl = np.ascontiguousarray(seq_lens, dtype=np.int32)
    dk = np.full(wl.dst_shape(), fill, dtype=np.float64)
    dv = np.full(wl.dst_shape(), fill, dtype=np.float64)
    lm = _map_arr(wl.layer_map)
    d = dims_of(wl)
    k_c, v_c, w_c = (np.ascontiguousarray(a) for a in (src_k, src_v, blob))
    rc = _load().oracle_translate_full(ctypes.byref(d), _ptr(lm), _ptr(k_c), _ptr(v_c),
                                       _ptr(w_c), sl.size, _ptr(sl),
                                       _ptr(dk), _ptr(dv))
    if rc != 0:
        raise ValueError("oracle_translate_full: invalid arguments")
    return dk, dv


def sample_tokens(seq_lens, n_per_seq: int, seed: int = 1, tile: int = 128):
    """A fixed token sample that always includes each sequence's first and last
    position and the positions on either side of every ``tile`` boundary (the
    sample layout is test bookkeeping, not method arithmetic)."""
    rng = np.random.default_rng(seed)
    tb, ts = [], []
    for b, L in enumerate(seq_lens):
        if L <= 0:
            continue
        pos = {0, L - 1}
        for k in range(tile, L, tile * max(1, (L // tile) // 4 or 1)):
            pos.update({k - 1, k})
        extra = max(0, n_per_seq - len(pos))
        if extra:
            pos.update(rng.integers(0, L, size=extra).tolist())
        for s in sorted(pos):
            tb.append(b)
            ts.append(s)
    return np.asarray(tb, dtype=np.int32), np.asarray(ts, dtype=np.int32)


# ---- backbone translators (App. C.2) -------------------------------------------

def bt_dims_of(wl) -> OracleBtDims:
    return OracleBtDims(*wl.bt)


def layernorm(x, gamma=None, beta=None) -> np.ndarray:
    """Layer norm of a vector (eps 1e-5, biased variance)."""
    xv = np.ascontiguousarray(x, dtype=np.float64)
    y = np.empty_like(xv)
    g = None if gamma is None else np.ascontiguousarray(gamma, dtype=np.float64)
    b = None if beta is None else np.ascontiguousarray(beta, dtype=np.float64)
    _load().oracle_layernorm(xv.ctypes.data, xv.size, _ptr(g), _ptr(b), y.ctypes.data)
    return y


def bt_attention(q, k, v, heads: int) -> np.ndarray:
    """Multi-head attention of the rows of q over the rows of k, v ([P][d] each)."""
    q, k, v = (np.ascontiguousarray(a, dtype=np.float64) for a in (q, k, v))
    P, d = q.shape
    o = np.empty_like(q)
    if _load().oracle_bt_attention(P, d, heads, q.ctypes.data, k.ctypes.data, v.ctypes.data,
                                   o.ctypes.data) != 0:
        raise ValueError("oracle_bt_attention: invalid sizes")
    return o


def bt_blob_elems(wl) -> int:
    return int(_load().oracle_bt_blob_elems(ctypes.byref(dims_of(wl)), ctypes.byref(bt_dims_of(wl))))


def bt_backbone(wl, blob, X: int, m: int, x):
    """One backbone translator (expert m of block X) on one token's window
    x[N][P][d_s]. Returns (Y[N][D_t], h[N][P][d])."""
    _, N, d, _, _ = wl.bt
    xv = np.ascontiguousarray(x, dtype=np.float64)
    y = np.empty((N, wl.d_tgt))
    h = np.empty((N, wl.src_kv_heads, d))
    w_c = np.ascontiguousarray(blob)
    rc = _load().oracle_bt_backbone(ctypes.byref(dims_of(wl)), ctypes.byref(bt_dims_of(wl)),
                                    _ptr(w_c), X, m, xv.ctypes.data,
                                    y.ctypes.data, h.ctypes.data)
    if rc != 0:
        raise ValueError("oracle_bt_backbone: invalid arguments")
    return y, h


def bt_tokens(wl, src_k, src_v, blob, tok_b, tok_s, gate_fixed=None, want_gate=False):
    """Backbone-translator MoT for sampled tokens. Returns out[N][2][n][D_t]
    (slot r = target layer window start + r) and, with ``want_gate``, the kept
    renormalised gate [2][n][E]."""
    tb = np.ascontiguousarray(tok_b, dtype=np.int32)
    ts = np.ascontiguousarray(tok_s, dtype=np.int32)
    n = tb.size
    N = wl.bt[1]
    out = np.full((N, 2, n, wl.d_tgt), np.nan)
    gate = np.full((2, n, wl.n_translators), np.nan) if want_gate else None
    gf = None if gate_fixed is None else np.ascontiguousarray(gate_fixed, dtype=np.float64)
    lm = _map_arr(wl.layer_map)
    k_c, v_c, w_c = (np.ascontiguousarray(a) for a in (src_k, src_v, blob))
    rc = _load().oracle_bt_tokens(ctypes.byref(dims_of(wl)), ctypes.byref(bt_dims_of(wl)),
                                  _ptr(lm), _ptr(k_c), _ptr(v_c), _ptr(w_c),
                                  n, _ptr(tb), _ptr(ts), _ptr(gf), _ptr(out), _ptr(gate))
    if rc != 0:
        raise ValueError("oracle_bt_tokens: invalid arguments")
    return (out, gate) if want_gate else out


# ---- replay attention (App. C.4) ---------------------------------------------------

def replay_dims_of(wl) -> OracleReplayDims:
    return OracleReplayDims(wl.max_batch, wl.max_seq, wl.q_heads, wl.kv_heads, wl.head_dim,
                            wl.top_s, wl.n_full)


def replay_select(wl, guide, b: int, u: int) -> np.ndarray:
    """Top-S positions (ascending) of row u of batch entry b's guidance map."""
    g = np.ascontiguousarray(guide)
    out = np.empty(min(wl.top_s, u + 1), dtype=np.int32)
    n = _load().oracle_replay_select(ctypes.byref(replay_dims_of(wl)), g.ctypes.data, b, u,
                                     out.ctypes.data)
    if n < 0:
        raise ValueError("oracle_replay_select: invalid arguments")
    return out[:n]


def replay_tokens(wl, layer: int, q, k, v, guide, tb, th, tu) -> np.ndarray:
    """Replay attention outputs [n][d] for queries (tb, th, tu) of target layer `layer`."""
    tb, th, tu = (np.ascontiguousarray(x, dtype=np.int32) for x in (tb, th, tu))
    q_c, k_c, v_c = (np.ascontiguousarray(a) for a in (q, k, v))
    g_c = None if guide is None else np.ascontiguousarray(guide)
    out = np.empty((tb.size, wl.head_dim))
    rc = _load().oracle_replay_tokens(ctypes.byref(replay_dims_of(wl)), layer, q_c.ctypes.data,
                                      k_c.ctypes.data, v_c.ctypes.data, _ptr(g_c), tb.size,
                                      tb.ctypes.data, th.ctypes.data, tu.ctypes.data,
                                      out.ctypes.data)
    if rc != 0:
        raise ValueError("oracle_replay_tokens: invalid arguments")
    return out
