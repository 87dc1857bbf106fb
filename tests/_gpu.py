"""Shared GPU-test plumbing: device buffers, one translation through the C ABI,
comparisons against the oracle. Imported only by tests marked ``gpu``."""
import numpy as np
import torch

from paper_2607_28979_gb300 import build as mot_build

mot_build.build()
import paper_2607_28979_gb300.mot as M   # noqa: E402

# Fill patterns for positions the translation must not touch.
SENTINEL_BF16 = 0x7F7F           # bf16 bits of a large finite value
SENTINEL_F32 = 0x7F7F7F7F
CANARY_ELEMS = 4096               # guard elements after the end of every dst buffer

# Parity bars (element-wise against the fp64 oracle).
TOL = {"bf16": dict(rel_rms=1e-2, max_abs=3e-2), "fp32": dict(rel_rms=1e-5, max_abs=1e-5)}


def to_device(wl, arr):
    if wl.dtype == "bf16":
        return torch.from_numpy(np.ascontiguousarray(arr).view(np.int16)).cuda().view(torch.bfloat16)
    return torch.from_numpy(np.ascontiguousarray(arr)).cuda()


def int_view(t):
    return t.view(torch.int16) if t.dtype == torch.bfloat16 else t.view(torch.int32)


def sentinel(wl):
    return SENTINEL_BF16 if wl.dtype == "bf16" else SENTINEL_F32


def alloc_dst(wl, lead=0):
    """A target cache with CANARY_ELEMS guard elements after its end and `lead`
    before its start (which shifts its alignment), all filled with the sentinel.
    Returns (full buffer, cache view)."""
    n = int(np.prod(wl.dst_shape()))
    dt = torch.bfloat16 if wl.dtype == "bf16" else torch.float32
    buf = torch.empty(lead + n + CANARY_ELEMS, dtype=dt, device="cuda")
    s = sentinel(wl)
    int_view(buf).fill_(s - (1 << 16) if wl.dtype == "bf16" and s >= 1 << 15 else s)
    return buf, buf[lead:lead + n].view(wl.dst_shape())


def sentinel_value(wl):
    s = sentinel(wl)
    return s - (1 << 16) if wl.dtype == "bf16" and s >= 1 << 15 else s


class Run:
    """One handle plus device inputs/outputs for a workload."""

    def __init__(self, wl, sk, sv, blob, seq_lens=None, batch=None, dst_lead=0):
        self.wl = wl
        self.h = M.mot_create(M.config_from(wl))
        M.mot_load_weights(self.h, blob)
        self.sk = to_device(wl, sk)
        self.sv = to_device(wl, sv)
        self.seq = list(wl.seq_lens if seq_lens is None else seq_lens)
        self.batch = len(self.seq) if batch is None else batch
        self.lens = torch.tensor(self.seq + [0] * max(0, 1 - len(self.seq)), dtype=torch.int32,
                                 device="cuda")
        self.lead = dst_lead
        self.buf_k, self.dk = alloc_dst(wl, dst_lead)
        self.buf_v, self.dv = alloc_dst(wl, dst_lead)

    def translate(self, stream=None):
        M.mot_translate(self.h, self.sk, self.sv, self.lens, self.batch, self.dk, self.dv, stream)
        return M.mot_get_device_status(self.h, stream)

    def canaries_intact(self):
        n, a = self.dk.numel(), self.lead
        s = sentinel_value(self.wl)
        return all(bool((int_view(b[a + n:]) == s).all()) and bool((int_view(b[:a]) == s).all())
                   for b in (self.buf_k, self.buf_v))

    def padding_untouched(self, lens=None):
        """Every position that must keep its contents still holds the sentinel."""
        wl, s = self.wl, sentinel_value(self.wl)
        lens = self.seq if lens is None else lens
        tl = set(wl.translated_layers())
        for dst in (self.dk, self.dv):
            iv = int_view(dst)
            for l in range(wl.n_layers_tgt):
                for b in range(wl.max_batch):
                    L = lens[b] if (l in tl and b < self.batch) else 0
                    L = max(0, min(L, wl.max_seq))
                    if not bool((iv[l, b, :, L:, :] == s).all()):
                        return False
        return True

    def dst_f64(self):
        return (self.dk.double().cpu().numpy(), self.dv.double().cpu().numpy())

    def gather(self, tb, ts):
        """GPU output rows at sampled tokens: [L_t][2][n][D_t] float64."""
        tb_t = torch.as_tensor(tb, dtype=torch.long, device="cuda")
        ts_t = torch.as_tensor(ts, dtype=torch.long, device="cuda")
        out = []
        for dst in (self.dk, self.dv):
            g = dst[:, tb_t, :, ts_t, :]           # [n, L_t, H_t, d_t] (advanced dims first)
            g = g.permute(1, 0, 2, 3).reshape(self.wl.n_layers_tgt, len(tb), -1)
            out.append(g.double().cpu().numpy())
        return np.stack(out, axis=1)


def metrics(got, ref):
    got = np.asarray(got, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    diff = got - ref
    rel_rms = float(np.sqrt((diff ** 2).sum() / max((ref ** 2).sum(), 1e-300)))
    max_abs = float(np.abs(diff).max()) if diff.size else 0.0
    return dict(rel_rms=rel_rms, max_abs=max_abs, max_ref=float(np.abs(ref).max()) if ref.size else 0.0,
                n=int(ref.size))


def assert_parity(wl, got, ref, label=""):
    m = metrics(got, ref)
    tol = TOL[wl.dtype]
    assert np.isfinite(got).all(), f"{label}: non-finite output"
    assert m["rel_rms"] <= tol["rel_rms"] and m["max_abs"] <= tol["max_abs"], f"{label}: {m} vs {tol}"
    return m


def translated_mask_full(wl, seq_lens, batch=None):
    """Boolean mask over the target-cache shape of the positions that are translated."""
    mask = np.zeros(wl.dst_shape(), dtype=bool)
    batch = len(seq_lens) if batch is None else batch
    for l in wl.translated_layers():
        for b in range(batch):
            mask[l, b, :, :max(0, min(seq_lens[b], wl.max_seq)), :] = True
    return mask
