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
