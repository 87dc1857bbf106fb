"""Test-side helpers: structured weight blobs and storage conversions.

These only lay numbers out in the library's documented blob order and convert
storage types; they implement none of the translation arithmetic.
"""
import numpy as np

import synth


def f32_to_bf16_bits(a):
    """Round fp32 values to bf16 bit patterns (round-to-nearest-even)."""
    u = np.ascontiguousarray(a, dtype=np.float32).view(np.uint32).astype(np.uint64)
    u = (u + 0x7FFF + ((u >> 16) & 1)) >> 16
    return u.astype(np.uint16)


def bf16_bits_to_f64(a):
    return (np.asarray(a, dtype=np.uint16).astype(np.uint32) << 16).view(np.float32).astype(np.float64)


def storage_to_f64(wl, a):
    return bf16_bits_to_f64(a) if wl.dtype == "bf16" else np.asarray(a, dtype=np.float64)


def to_storage(wl, a):
    a = np.asarray(a, dtype=np.float64)
    if wl.dtype == "bf16":
        return f32_to_bf16_bits(a.astype(np.float32))
    return a.astype(np.float32)


def make_blob(wl, group_fn):
    """Blob for ``wl`` whose (layer l, x) block comes from ``group_fn(l, x)``, a dict
    with Wg[E][Ds], bg[E], W1[E][H][Ds], b1[E][H], W2[E][Dt][H], b2[E][Dt]."""
    parts = []
    for l in wl.translated_layers():
        for x in (0, 1):
            g = group_fn(l, x)
            parts += [np.ravel(g["Wg"]), np.ravel(g["bg"])]
            for m in range(wl.n_translators):
                parts += [np.ravel(g["W1"][m]), np.ravel(g["b1"][m]),
                          np.ravel(g["W2"][m]), np.ravel(g["b2"][m])]
    flat = np.concatenate(parts) if parts else np.zeros(0)
    assert flat.size == wl.blob_elems()
    return to_storage(wl, flat)


def split_blob(wl, blob):
    """Inverse of make_blob: {(l, x): dict of fp64 arrays}."""
    f = storage_to_f64(wl, blob)
    E, Ds, Dt, H = wl.n_translators, wl.d_src, wl.d_tgt, wl.hidden
    out = {}
    for (l, x, t, m, off, n, _) in synth.blob_offsets(wl):
        g = out.setdefault((l, x), {"W1": [None] * E, "b1": [None] * E,
                                    "W2": [None] * E, "b2": [None] * E})
        a = f[off:off + n]
        if t == synth.T_WG:
            g["Wg"] = a.reshape(E, Ds)
        elif t == synth.T_BG:
            g["bg"] = a
        elif t == synth.T_W1:
            g["W1"][m] = a.reshape(H, Ds)
        elif t == synth.T_B1:
            g["b1"][m] = a
        elif t == synth.T_W2:
            g["W2"][m] = a.reshape(Dt, H)
        else:
            g["b2"][m] = a
    return out


def signed_perm_translator(D, H, perm_in, perm_out, scale=1.0, b_in=None, b_out=None):
    """One translator whose output is scale * (Q (P z + b_in)) + b_out exactly.

    W1 = [P; -P] (zero-padded to H rows), b1 = [b_in; -b_in], W2 = scale*[Q, -Q],
    using GELU(x) - GELU(-x) = x for every x."""
    assert H >= 2 * D
    P = np.zeros((D, D)); P[np.arange(D), perm_in] = 1.0
    Q = np.zeros((D, D)); Q[np.arange(D), perm_out] = 1.0
    W1 = np.zeros((H, D)); W1[:D] = P; W1[D:2 * D] = -P
    b1 = np.zeros(H)
    if b_in is not None:
        b1[:D] = b_in; b1[D:2 * D] = -np.asarray(b_in)
    W2 = np.zeros((D, H)); W2[:, :D] = scale * Q; W2[:, D:2 * D] = -scale * Q
    b2 = np.zeros(D) if b_out is None else np.asarray(b_out, dtype=np.float64)
    return W1, b1, W2, b2


def gather_src(wl, src, layer, b, s):
    """Source vector z of token (b, s) at source layer ``layer``: head-major flatten."""
    return storage_to_f64(wl, src[layer, b, :, s, :]).reshape(-1)


def dst_row(dst, l, b, s):
    """Target vector at (layer l, b, s) from a target-layout cache, head-major."""
    return np.asarray(dst[l, b, :, s, :]).reshape(-1)


def stratified_tokens(seq_lens, n_random, seed=1, tile=128):
    """A token sample spread over the batch: n_random positions split across the
    sequences in proportion to their lengths, always including each sequence's
    first and last position and the positions on either side of some `tile`
    boundaries. Returns (tb, ts) int32 arrays (test bookkeeping only)."""
    rng = np.random.default_rng(seed)
    total = sum(max(0, L) for L in seq_lens)
    tb, ts = [], []
    for b, L in enumerate(seq_lens):
        if L <= 0:
            continue
        k = min(L, max(2, int(round(n_random * L / max(total, 1)))))
        pos = {0, L - 1}
        bounds = list(range(tile, L, tile))
        for t in rng.permutation(bounds)[:max(1, k // 8)] if bounds else []:
            pos.update({int(t) - 1, int(t)})
        for p in rng.permutation(L).tolist():   # random positions until k are chosen
            if len(pos) >= k:
                break
            pos.add(p)
        pos = sorted(pos)
        tb += [b] * len(pos)
        ts += pos
    return np.asarray(tb, dtype=np.int32), np.asarray(ts, dtype=np.int32)


def whole_tiles(seq_lens, tile=256, seed=2, last=True):
    """Every token of one `tile`-aligned window per sequence (the rows of one
    tile of the tensor-core schedule), plus, with `last`, the final window of the
    last non-empty sequence (the last wave of a persistent schedule). A sequence
    shorter than `tile` contributes all its tokens."""
    rng = np.random.default_rng(seed)
    tb, ts = [], []
    seen = set()
    for b, L in enumerate(seq_lens):
        if L <= 0:
            continue
        n_win = max(1, L // tile)
        w = int(rng.integers(0, n_win))
        seen.add((b, w))
        s0 = w * tile
        for s in range(s0, min(L, s0 + tile)):
            tb.append(b)
            ts.append(s)
    if last:
        nz = [b for b, L in enumerate(seq_lens) if L > 0]
        if nz:
            b = nz[-1]
            L = seq_lens[b]
            w = max(0, (L - 1) // tile)
            if (b, w) not in seen:
                for s in range(w * tile, L):
                    tb.append(b)
                    ts.append(s)
    return np.asarray(tb, dtype=np.int32), np.asarray(ts, dtype=np.int32)


def restrict_layers(wl, blob, layer_map, keep):
    """The workload and blob for computing only target layers `keep` (the other
    target layers marked untranslated): each kept layer's blocks (K and V, or
    the one MoT-h block) are cut out of the full blob, in blob order. `layer_map` is the full map in use."""
    tl = [l for l in range(wl.n_layers_tgt) if layer_map[l] >= 0]
    gsz = wl.group_elems()
    nx = 1 if wl.is_h else 2   # MoT-h: one block per layer
    parts = []
    for r, l in enumerate(tl):
        if l in keep:
            parts.append(blob[nx * r * gsz:nx * (r + 1) * gsz])
    lm = tuple(layer_map[l] if l in keep else -1 for l in range(wl.n_layers_tgt))
    return wl.replace(layer_map=lm), np.concatenate(parts)
