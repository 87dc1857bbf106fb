"""Seeded synthetic workloads for the MoT KV-cache translation pass.

This package draws the inputs that both the fp64 oracle and the CUDA path
consume: source K/V caches, the packed translator weight blob and the ragged
sequence lengths. It holds none of the translation method's arithmetic (no
gate, GELU, layer mapping or combine) -- only random draws, storage rounding
and the blob's byte layout, which is part of the library interface.

Value recipe (stands in for real model caches and trained translators, which
are not available):
  * K, V = s_c * N(0, 1), with a per-channel scale s_c ~ LogNormal(0, 0.5)
    drawn once per (source layer, K/V, channel c = h*d + i);
  * every weight and bias ~ N(0, 1/fan_in): fan_in = D_s for the gate and the
    first translator layer, H for the second (backbone translators: the input
    width of each linear map);
  * backbone layer norms: gain ~ 1 + 0.1 N(0, 1), shift ~ 0.1 N(0, 1);
  * fp64 draws rounded to fp32, then (bf16 workloads) to bf16 with
    round-to-nearest-even.

The generator itself (SplitMix64 + Box-Muller) is implemented in ``synth.c``.
"""
from __future__ import annotations

import ctypes
import dataclasses
import os
import subprocess
from typing import Optional, Sequence, Tuple

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "synth.c")
_LIB = os.path.join(_HERE, "libsynth.so")

# Blob tensor ids, in blob order within one (target layer, K/V) group.
T_WG, T_BG, T_W1, T_B1, T_W2, T_B2, T_WK, T_WV = range(8)

# Backbone-translator blob tensors (App. C.2), in blob order: the window gate,
# then per expert the input block, per slot one CAB block, then the output block.
BT_TENSORS = ("wg", "bg", "lnin_g", "lnin_b", "win", "bin",
              "lnq_g", "lnq_b", "lnc_g", "lnc_b", "wq", "bq", "wk", "bk", "wv", "bv", "wo", "bo",
              "lnf_g", "lnf_b", "wf1", "bf1", "wf2", "bf2",
              "lnout_g", "lnout_b", "wout", "bout")
BT_ID = {name: 16 + i for i, name in enumerate(BT_TENSORS)}


def build(force: bool = False) -> str:
    """Compile ``libsynth.so`` next to its source if it is missing or stale."""
    if force or not os.path.exists(_LIB) or os.path.getmtime(_LIB) < os.path.getmtime(_SRC):
        tmp = _LIB + f".{os.getpid()}.tmp"
        subprocess.check_call(
            ["gcc", "-O2", "-fopenmp", "-shared", "-fPIC", "-o", tmp, _SRC, "-lm"])
        os.replace(tmp, _LIB)
    return _LIB


_lib = None


def _load():
    global _lib
    if _lib is None:
        lib = ctypes.CDLL(build())
        lib.synth_stream_key.restype = ctypes.c_uint64
        lib.synth_stream_key.argtypes = [ctypes.c_uint64, ctypes.c_uint64]
        lib.synth_splitmix64.restype = ctypes.c_uint64
        lib.synth_splitmix64.argtypes = [ctypes.c_uint64, ctypes.c_uint64]
        lib.synth_normal_at.restype = ctypes.c_double
        lib.synth_normal_at.argtypes = [ctypes.c_uint64, ctypes.c_uint64]
        lib.synth_fill_normal.restype = None
        lib.synth_fill_normal.argtypes = [ctypes.c_uint64, ctypes.c_uint64, ctypes.c_int64,
                                          ctypes.c_double, ctypes.c_int, ctypes.c_void_p]
        lib.synth_fill_normal_shifted.restype = None
        lib.synth_fill_normal_shifted.argtypes = [ctypes.c_uint64, ctypes.c_uint64, ctypes.c_int64,
                                                  ctypes.c_double, ctypes.c_double, ctypes.c_int,
                                                  ctypes.c_void_p]
        lib.synth_fill_guide.restype = None
        lib.synth_fill_guide.argtypes = [ctypes.c_uint64, ctypes.c_uint64, ctypes.c_int,
                                         ctypes.c_int, ctypes.c_int, ctypes.c_void_p]
        lib.synth_fill_cache_layer.restype = None
        lib.synth_fill_cache_layer.argtypes = [ctypes.c_uint64, ctypes.c_uint64, ctypes.c_uint64,
                                               ctypes.c_int, ctypes.c_int, ctypes.c_int,
                                               ctypes.c_int, ctypes.c_int, ctypes.c_void_p]
        _lib = lib
    return _lib


@dataclasses.dataclass(frozen=True)
class Workload:
    """Shapes of one translation workload (mirrors the C ``mot_config``)."""
    name: str
    n_layers_src: int
    src_kv_heads: int
    src_head_dim: int
    n_layers_tgt: int
    tgt_kv_heads: int
    tgt_head_dim: int
    n_translators: int
    hidden: int
    max_batch: int
    max_seq: int
    dtype: str                      # "bf16" or "fp32"
    seq_lens: Tuple[int, ...]
    top_k: int = 0                  # 0 (or E) = dense softmax gate
    layer_map: Optional[Tuple[int, ...]] = None   # None = depth-ratio default; -1 = untranslated
    # MoT-h (App. C.5): > 0 = the target activation width d_at. The source tensor is
    # then the activation [L_s][B][S][d_as], stored as a one-head cache
    # (src_kv_heads = 1, src_head_dim = d_as); the target caches are restored
    # through per-layer projections W^K, W^V [D_t][d_at].
    act_tgt: int = 0
    # Backbone translators (App. C.2): (window start, window length N, width d,
    # attention heads n_a, FFN width d_f). The window is target layers
    # start .. start+N-1; each source-head row of a slot is one attention row.
    bt: Optional[Tuple[int, int, int, int, int]] = None

    @property
    def is_bt(self) -> bool:
        return self.bt is not None

    @property
    def bt_window(self) -> list:
        q, n = self.bt[0], self.bt[1]
        return list(range(q, q + n))

    @property
    def d_src(self) -> int:
        return self.src_kv_heads * self.src_head_dim

    @property
    def d_tgt(self) -> int:
        return self.tgt_kv_heads * self.tgt_head_dim

    @property
    def batch(self) -> int:
        return len(self.seq_lens)

    @property
    def tokens(self) -> int:
        return int(sum(self.seq_lens))

    @property
    def np_dtype(self):
        return np.uint16 if self.dtype == "bf16" else np.float32

    @property
    def esize(self) -> int:
        return 2 if self.dtype == "bf16" else 4

    def translated_layers(self) -> list:
        """Target layers that receive a translation (all, unless the map says -1)."""
        if self.layer_map is None:
            return list(range(self.n_layers_tgt))
        return [l for l, s in enumerate(self.layer_map) if s >= 0]

    def src_shape(self):
        return (self.n_layers_src, self.max_batch, self.src_kv_heads, self.max_seq, self.src_head_dim)

    def dst_shape(self):
        return (self.n_layers_tgt, self.max_batch, self.tgt_kv_heads, self.max_seq, self.tgt_head_dim)

    @property
    def is_h(self) -> bool:
        return self.act_tgt > 0

    @property
    def d_mix(self) -> int:
        """Output width of the translator mixture: D_t, or d_at for MoT-h."""
        return self.act_tgt if self.is_h else self.d_tgt

    def group_elems(self) -> int:
        """Elements of one block of the weight blob: a (target layer, K/V) group,
        or for MoT-h a target layer (mixture, then W^K and W^V), or for backbone
        translators a K/V block (window gate, then every expert)."""
        if self.is_bt:
            return sum(item[5] for item in bt_blob_offsets(self) if item[0] == 0)
        E, Ds, Dm, H = self.n_translators, self.d_src, self.d_mix, self.hidden
        n = E * Ds + E + E * (H * Ds + H + Dm * H + Dm)
        return n + (2 * self.d_tgt * self.act_tgt if self.is_h else 0)

    def blob_elems(self) -> int:
        if self.is_bt:
            return 2 * self.group_elems()
        return (1 if self.is_h else 2) * len(self.translated_layers()) * self.group_elems()

    def replace(self, **kw) -> "Workload":
        return dataclasses.replace(self, **kw)


# The five workloads: shapes of the paper's model pairs.
WORKLOADS = {
    # GPT-2-small (first 4 layers, 12x64) -> OPT-125m-shaped (4 layers, 12x64), fp32.
    "tiny_fp32": Workload("tiny_fp32", 4, 12, 64, 4, 12, 64, 2, 768, 1, 64, "fp32", (64,)),
    # GPT-2-small -> OPT-125m, 12 layers each, E=4, MLP 768->1536->768.
    "gpt2s_opt125m": Workload("gpt2s_opt125m", 12, 12, 64, 12, 12, 64, 4, 1536, 8, 1024, "bf16",
                              (1024,) * 8),
    # Qwen2.5-0.5B (24L, 2x64) -> Qwen2.5-1.5B (28L, 2x128), E=4, MLP 128->1024->256.
    "qwen05_qwen15": Workload("qwen05_qwen15", 24, 2, 64, 28, 2, 128, 4, 1024, 4, 4096, "bf16",
                              (4096,) * 4),
    # GPT-2-medium (24L, 16x64) -> Qwen2.5-7B (28L, 4x128), E=8, MLP 1024->2048->512.
    "gpt2m_qwen7": Workload("gpt2m_qwen7", 24, 16, 64, 28, 4, 128, 8, 2048, 2, 8192, "bf16",
                            (8192,) * 2),
    # Qwen2.5-7B -> Qwen2.5-7B (28L, 4x128), ragged batch of 4 long sequences.
    "qwen7_long": Workload("qwen7_long", 28, 4, 128, 28, 4, 128, 4, 2048, 4, 32768, "bf16",
                           (32768, 16384, 8192, 4096)),
}

# MoT-h (App. C.5) counterparts of two of the model pairs: the source activation
# is the model width (d_model) of the source model, the translated activation
# the target model's, and K, V are restored through the target's projections.
WORKLOADS.update({
    # GPT-2-small (768) -> OPT-125m (768; KV 12x64), 12 layers each, E=4, MLP 768->1536->768.
    "h_gpt2s_opt125m": Workload("h_gpt2s_opt125m", 12, 1, 768, 12, 12, 64, 4, 1536, 8, 1024,
                                "bf16", (1024,) * 8, act_tgt=768),
    # Qwen2.5-0.5B (896, 24L) -> Qwen2.5-1.5B (1536, 28L; KV 2x128), E=4, MLP 896->1024->1536.
    "h_qwen05_qwen15": Workload("h_qwen05_qwen15", 24, 1, 896, 28, 2, 128, 4, 1024, 4, 4096,
                                "bf16", (4096,) * 4, act_tgt=1536),
})

# Backbone-translator (App. C.2) counterparts: a channel window of about 0.3 of
# the layers (the paper's default ratio), N_Tr = 2 backbones with Top-1 routing
# (the paper's default (Top-K, N_Tr) = (1, 2)), rows of width 128 with 4
# attention heads and an FFN of 512.
WORKLOADS.update({
    # GPT-2-small -> OPT-125m (12x64 -> 12x64): window = target layers 4..7.
    "bt_gpt2s_opt125m": Workload("bt_gpt2s_opt125m", 12, 12, 64, 12, 12, 64, 2, 0, 8, 1024,
                                 "bf16", (1024,) * 8, top_k=1, bt=(4, 4, 128, 4, 512)),
    # Qwen2.5-0.5B (24L, 2x64) -> Qwen2.5-1.5B (28L, 2x128): window = target layers 10..17.
    "bt_qwen05_qwen15": Workload("bt_qwen05_qwen15", 24, 2, 64, 28, 2, 128, 2, 0, 4, 4096,
                                 "bf16", (4096,) * 4, top_k=1, bt=(10, 8, 128, 4, 512)),
})

# Order in which the workloads are listed in the build's benchmark configuration.
WORKLOAD_ORDER = ["tiny_fp32", "gpt2s_opt125m", "qwen05_qwen15", "gpt2m_qwen7", "qwen7_long"]


def _stream_cache(kind: int, x: int, layer: int) -> int:
    return (kind << 56) | (x << 48) | layer


def _stream_weight(layer: int, x: int, expert: int, tensor: int) -> int:
    return (3 << 56) | (x << 48) | (layer << 24) | (expert << 8) | tensor


def gen_cache(wl: Workload, x: int, seed: int = 0) -> np.ndarray:
    """Source cache for K (x=0) or V (x=1): [L_s][B][H_s][S_max][d_s] in storage dtype."""
    lib = _load()
    shape = wl.src_shape()
    out = np.empty(shape, dtype=wl.np_dtype)
    dt = 0 if wl.dtype == "bf16" else 1
    for l in range(wl.n_layers_src):
        view = out[l]
        lib.synth_fill_cache_layer(seed, _stream_cache(1, x, l), _stream_cache(2, x, l),
                                   wl.max_batch, wl.src_kv_heads, wl.max_seq, wl.src_head_dim,
                                   dt, view.ctypes.data)
    return out


def blob_offsets(wl: Workload):
    """Yield (target layer, x, tensor id, expert, offset, numel, fan_in) for every blob tensor."""
    E, Ds, Dt, H, Dm = wl.n_translators, wl.d_src, wl.d_tgt, wl.hidden, wl.d_mix
    off = 0
    for l in wl.translated_layers():
        for x in ((0,) if wl.is_h else (0, 1)):
            yield (l, x, T_WG, 0, off, E * Ds, Ds); off += E * Ds
            yield (l, x, T_BG, 0, off, E, Ds); off += E
            for m in range(E):
                yield (l, x, T_W1, m, off, H * Ds, Ds); off += H * Ds
                yield (l, x, T_B1, m, off, H, Ds); off += H
                yield (l, x, T_W2, m, off, Dm * H, H); off += Dm * H
                yield (l, x, T_B2, m, off, Dm, H); off += Dm
            if wl.is_h:   # the target's key and value projections of layer l
                yield (l, x, T_WK, 0, off, Dt * Dm, Dm); off += Dt * Dm
                yield (l, x, T_WV, 0, off, Dt * Dm, Dm); off += Dt * Dm


def bt_blob_offsets(wl: Workload):
    """Backbone-translator blob: yield (x, name, expert, slot, offset, numel, mean, std)
    for every tensor, in blob order (slot -1 = not a CAB tensor)."""
    E, P, ds, Ds, Dt = wl.n_translators, wl.src_kv_heads, wl.src_head_dim, wl.d_src, wl.d_tgt
    _, N, d, _, df = wl.bt
    off = 0

    def t(x, name, m, r, n, fan_in=None):
        nonlocal off
        if name.endswith("_g"):
            mean, std = 1.0, 0.1
        elif name.startswith("ln"):
            mean, std = 0.0, 0.1
        else:
            mean, std = 0.0, 1.0 / np.sqrt(fan_in)
        item = (x, name, m, r, off, n, mean, std)
        off += n
        return item

    for x in (0, 1):
        yield t(x, "wg", 0, -1, E * N * Ds, N * Ds)
        yield t(x, "bg", 0, -1, E, N * Ds)
        for m in range(E):
            yield t(x, "lnin_g", m, -1, ds)
            yield t(x, "lnin_b", m, -1, ds)
            yield t(x, "win", m, -1, d * ds, ds)
            yield t(x, "bin", m, -1, d, ds)
            for r in range(N):
                for nm in ("lnq_g", "lnq_b", "lnc_g", "lnc_b"):
                    yield t(x, nm, m, r, d)
                for nm in ("wq", "wk", "wv", "wo"):
                    yield t(x, nm, m, r, d * d, d)
                    yield t(x, "b" + nm[1], m, r, d, d)
                yield t(x, "lnf_g", m, r, d)
                yield t(x, "lnf_b", m, r, d)
                yield t(x, "wf1", m, r, df * d, d)
                yield t(x, "bf1", m, r, df, d)
                yield t(x, "wf2", m, r, d * df, df)
                yield t(x, "bf2", m, r, d, df)
            yield t(x, "lnout_g", m, -1, P * d)
            yield t(x, "lnout_b", m, -1, P * d)
            yield t(x, "wout", m, -1, Dt * P * d, P * d)
            yield t(x, "bout", m, -1, Dt, P * d)


def gen_weights(wl: Workload, seed: int = 0) -> np.ndarray:
    """Packed weight blob (flat, storage dtype) in the library's documented order."""
    lib = _load()
    out = np.empty(wl.blob_elems(), dtype=wl.np_dtype)
    dt = 0 if wl.dtype == "bf16" else 1
    base = out.ctypes.data
    if wl.is_bt:
        end = 0
        for (x, name, m, r, off, n, mean, std) in bt_blob_offsets(wl):
            stream = _stream_weight(r & 0xFFFF, x, m, BT_ID[name])
            lib.synth_fill_normal_shifted(seed, stream, n, mean, std, dt, base + off * wl.esize)
            end = off + n
        assert end == out.size
        return out
    for (l, x, t, m, off, n, fan_in) in blob_offsets(wl):
        lib.synth_fill_normal(seed, _stream_weight(l, x, m, t), n, 1.0 / np.sqrt(fan_in), dt,
                              base + off * wl.esize)
    assert off + n == out.size
    return out


def seq_lens_array(wl: Workload) -> np.ndarray:
    return np.asarray(wl.seq_lens, dtype=np.int32)


def normal(seed: int, stream: int, n: int) -> np.ndarray:
    """n fp64 standard-normal draws of one stream (for tests of the generator)."""
    out = np.empty(n, dtype=np.float64)
    _load().synth_fill_normal(seed, stream, n, 1.0, 2, out.ctypes.data)
    return out


def splitmix64(key: int, n: int) -> int:
    return int(_load().synth_splitmix64(key, n))


def stream_key(seed: int, stream: int) -> int:
    return int(_load().synth_stream_key(seed, stream))


# ---- replay attention (App. C.4) -------------------------------------------------

@dataclasses.dataclass(frozen=True)
class ReplayWorkload:
    """One replay pass over the target model's layers: per layer the queries
    [B][Hq][N][d], the replay cache [B][Hkv][N][d] and, for layers >= n_full,
    the head-averaged guidance map [B][N][N] of source layer pi(l) (depth-ratio
    map from the source's n_layers_src layers)."""
    name: str
    n_layers_src: int
    n_layers_tgt: int
    q_heads: int
    kv_heads: int
    head_dim: int
    max_batch: int
    max_seq: int
    seq_lens: Tuple[int, ...]
    top_s: int = 128
    n_full: int = 2
    dtype: str = "bf16"

    @property
    def batch(self) -> int:
        return len(self.seq_lens)

    @property
    def tokens(self) -> int:
        return int(sum(self.seq_lens))

    def replace(self, **kw) -> "ReplayWorkload":
        return dataclasses.replace(self, **kw)


REPLAY_WORKLOADS = {
    # Qwen2.5-0.5B (24 layers) guiding Qwen2.5-1.5B (28 layers, 12 query heads, 2 KV heads
    # of 128), a 4K-token context budget (the paper's smallest long-context budget), S = 128,
    # L_Full = 2 (the paper's settings).
    "replay_qwen05_qwen15": ReplayWorkload("replay_qwen05_qwen15", 24, 28, 12, 2, 128, 4, 4096,
                                           (4096,) * 4),
}


def _stream_replay(kind: int, layer: int) -> int:
    return (4 << 56) | (kind << 48) | layer


def gen_replay_qkv(wl: ReplayWorkload, layer: int, seed: int = 0):
    """(q, k, v) of one target layer in bf16 bits: N(0, 1) draws."""
    lib = _load()
    B, N, d = wl.max_batch, wl.max_seq, wl.head_dim
    out = []
    for kind, H in ((1, wl.q_heads), (2, wl.kv_heads), (3, wl.kv_heads)):
        a = np.empty((B, H, N, d), dtype=np.uint16)
        lib.synth_fill_normal(seed, _stream_replay(kind, layer), a.size, 1.0, 0, a.ctypes.data)
        out.append(a)
    return tuple(out)


def gen_guide(wl: ReplayWorkload, src_layer: int, seed: int = 0) -> np.ndarray:
    """Guidance map of one source layer: [B][N][N] bf16 bits (zeros above the diagonal)."""
    a = np.empty((wl.max_batch, wl.max_seq, wl.max_seq), dtype=np.uint16)
    _load().synth_fill_guide(seed, _stream_replay(4, src_layer), wl.max_batch, wl.max_seq, 0,
                             a.ctypes.data)
    return a
