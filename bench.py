#!/usr/bin/env python3
"""Benchmark of the MoT KV-cache translation pass on GB300.

Metric: source-context tokens translated per second into the full target
cache (sum of seq_lens per mot_translate call, all translated layers, K and V).

One step = one mot_translate call over one synthetic batch of the workload,
with inputs resident in HBM. The default workload is the largest bf16 model
pair: Qwen2.5-7B-shaped -> Qwen2.5-7B-shaped caches (28 layers, 4 KV heads of
128), E=4 translators 512->2048->512, a ragged batch of 4 sequences of
32768/16384/8192/4096 tokens (61,440 tokens per step). Every step reads and
writes 8 GB (source caches, weights, target caches), far more than the
129 MB L2, so no flush is needed between steps. The same line carries, under
``per_config``, the device-resident timing of the other three bf16 model pairs
(GPT-2-small -> OPT-125m, Qwen2.5-0.5B -> 1.5B, GPT-2-medium -> Qwen2.5-7B),
each with its step roofline and its dominant kernel's fraction.

Roofline peaks: the burst bf16 figure applies when the run's own clock record
shows neither the power cap nor a lowered SM clock under load; otherwise the
sustained figure. Both fractions are printed.

  python bench.py [--gpus N --steps K --warmup W] [--impl mot|reference]

With N > 1 (torchrun) every rank runs an independent replica of the workload
(the translation shards by token and by layer with no exchange step); value is
all ranks' tokens over the slowest rank's time. ``--impl reference`` times the
fp64 CPU oracle on bounded token samples of the same workload.
"""
from __future__ import annotations

import argparse
import hashlib
import re
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import numpy as np   # noqa: E402

import synth   # noqa: E402

METRIC = "source-context tokens translated/sec into full target cache (1×GB300); % of roofline"
UNIT = "tokens/s"
DEFAULT_WORKLOAD = "qwen7_long"
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}


def workload_desc(wl) -> str:
    gate = ("dense softmax gate" if wl.top_k in (0, wl.n_translators)
            else f"softmax gate, Top-{wl.top_k} routing")
    if wl.is_bt:
        q, N, d, na, df = wl.bt
        return (f"{wl.name}: backbone translators (App. C.2), {wl.n_layers_src}L "
                f"{wl.src_kv_heads}x{wl.src_head_dim} -> {wl.n_layers_tgt}L "
                f"{wl.tgt_kv_heads}x{wl.tgt_head_dim}, window = target layers {q}..{q + N - 1}, "
                f"E={wl.n_translators} backbones (rows of width {d}, {na} heads over the "
                f"{wl.src_kv_heads} source heads, FFN {df}), {gate} on the window, {wl.dtype}, "
                f"batch {wl.batch} seq_lens {list(wl.seq_lens)}")
    if wl.is_h:
        return (f"{wl.name}: MoT-h, activations {wl.n_layers_src}L x {wl.src_head_dim} -> "
                f"{wl.n_layers_tgt}L x {wl.act_tgt}, E={wl.n_translators} MLP "
                f"{wl.src_head_dim}-{wl.hidden}-{wl.act_tgt} GELU, {gate}, K/V restored through "
                f"W^K, W^V to {wl.tgt_kv_heads}x{wl.tgt_head_dim}, {wl.dtype}, "
                f"batch {wl.batch} seq_lens {list(wl.seq_lens)}")
    return (f"{wl.name}: {wl.n_layers_src}L {wl.src_kv_heads}x{wl.src_head_dim} -> "
            f"{wl.n_layers_tgt}L {wl.tgt_kv_heads}x{wl.tgt_head_dim}, E={wl.n_translators} MLP "
            f"{wl.d_src}-{wl.hidden}-{wl.d_tgt} GELU, {gate}, {wl.dtype}, "
            f"batch {wl.batch} seq_lens {list(wl.seq_lens)}")


def algorithmic_bt(wl, layer_map):
    """FLOPs and bytes the backbone-translator method needs per step, and the
    FLOPs of each kernel per launch (one launch covers both K/V blocks and all
    backbones of one window slot)."""
    T, E, Ds, Dt, P, ds = (wl.tokens, wl.n_translators, wl.d_src, wl.d_tgt, wl.src_kv_heads,
                           wl.src_head_dim)
    q, N, d, na, df = wl.bt
    Ea = wl.top_k if 0 < wl.top_k < E else E
    rows = 2 * Ea * T * P            # (K/V, backbone, token, source head) rows of one slot
    per_launch = {
        "bt_in_ln_gelu": rows * 2 * ds * d,
        "bt_q": rows * 2 * d * d,
        "bt_kv": rows * 2 * d * 2 * d,
        "bt_attn": rows * P * 4 * d,
        "bt_o_residual_ln": rows * 2 * d * d,
        "bt_ffn1_gelu": rows * 2 * d * df,
        "bt_ffn2_residual_ln": rows * 2 * df * d,
        "bt_out_gelu_combine": 2 * Ea * T * 2 * P * d * Dt,
        "bt_gate": 2 * T * 2 * N * Ds * E,
    }
    per_launch["bt_ffn_fused"] = per_launch["bt_ffn1_gelu"] + per_launch["bt_ffn2_residual_ln"]
    flops = per_launch["bt_gate"] + N * sum(v for k, v in per_launch.items()
                                            if k not in ("bt_gate", "bt_ffn_fused"))
    # bytes each kernel must move per launch in this unfused schedule (its operand
    # rows in and result rows out; a slot after the first): its own HBM roofline
    es = wl.esize
    allrows = 2 * E * T * P
    bpl = {
        "bt_in_ln_gelu": 2 * E * T * Ds * es + allrows * d * 2,
        "bt_q": allrows * d * 2 * 2,
        "bt_kv": allrows * (d + 2 * d) * 2,
        "bt_attn": allrows * (3 * d + d) * 2,
        "bt_o_residual_ln": allrows * (d * 2 + d * 4 + d * 4 + d * 2),
        "bt_ffn1_gelu": allrows * (d + df) * 2,
        "bt_ffn2_residual_ln": allrows * (df * 2 + d * 4 + d * 4 + d * 2 + d * 2 + 8),
        "bt_out_gelu_combine": allrows * (d * 2 + 8) + 2 * T * Dt * es,
        "bt_gate": 2 * N * T * Ds * es,
        # FFN1 + GELU + FFN2 in one kernel: no hidden rows in HBM
        "bt_ffn_fused": allrows * (d * 2 + d * 4 + d * 4 + d * 2 + d * 2 + 8),
    }
    src_layers = {layer_map[t] for t in range(q, q + N)}
    bytes_src = 2 * len(src_layers) * T * Ds * es
    bytes_dst = 2 * N * T * Dt * es
    bytes_w = wl.blob_elems() * es
    return dict(flops=flops, per_launch=per_launch, bytes_per_launch=bpl,
                bytes=bytes_src + bytes_dst + bytes_w,
                bytes_src=bytes_src, bytes_dst=bytes_dst, bytes_w=bytes_w)


def algorithmic(wl, layer_map):
    """FLOPs and bytes the method needs per step (no intermediate traffic).
    ``layer_map``: the channel map in use (source layer per target layer, -1 = none)."""
    if wl.is_bt:
        return algorithmic_bt(wl, layer_map)
    T, E, Ds, Dt, Hh, Dm = wl.tokens, wl.n_translators, wl.d_src, wl.d_tgt, wl.hidden, wl.d_mix
    n_tl = len(wl.translated_layers())
    groups = n_tl if wl.is_h else 2 * n_tl   # MoT-h: one mixture per layer
    f_gate = 2 * Ds * E
    # with Top-K routing only the top_k chosen translators run on a token
    Ea = wl.top_k if 0 < wl.top_k < E else E
    f_g1 = Ea * 2 * Ds * Hh
    f_g2 = Ea * 2 * Hh * Dm + 2 * Ea * Dm
    f_proj = 2 * Dm * 2 * Dt if wl.is_h else 0   # MoT-h: K, V = W^K a_hat, W^V a_hat
    src_layers = {s for s in layer_map if s >= 0}
    es = wl.esize
    bytes_src = (1 if wl.is_h else 2) * len(src_layers) * T * Ds * es
    bytes_dst = 2 * n_tl * T * Dt * es
    bytes_w = wl.blob_elems() * es
    return dict(flops=groups * T * (f_gate + f_g1 + f_g2 + f_proj), flops_gemm1=groups * T * f_g1,
                flops_gemm2=groups * T * f_g2, flops_proj=groups * T * f_proj,
                bytes=bytes_src + bytes_dst + bytes_w,
                bytes_src=bytes_src, bytes_dst=bytes_dst, bytes_w=bytes_w)


def load_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return d, "measured"
    return FALLBACK_PEAKS, "fallback"


# Source files each profiled kernel is built from (its traffic figure is stale
# once any of them changes).
KERNEL_SOURCES = {
    "umma2_gemm1_gelu_gate": ["umma2.cu", "umma_common.cuh", "gelu.cuh", "ptx.cuh",
                              "mot_internal.h"],
    "umma2_gemm2_combine_store": ["umma2.cu", "umma_common.cuh", "gelu.cuh", "ptx.cuh",
                                  "mot_internal.h"],
    "umma2_onchip_translate": ["onchip.cu", "umma_common.cuh", "gelu.cuh", "ptx.cuh",
                               "mot_internal.h"],
    "umma2_wide_translate": ["wide.cu", "umma_common.cuh", "gelu.cuh", "ptx.cuh", "mot_internal.h"],
    # replay stages: guided attention, selection (with the SIMT kernels), full attention
    "replay_attn_sparse": ["replay_gattn.cu", "replay_common.cuh", "replay_internal.h",
                           "mot_internal.h", "ptx.cuh"],
    "replay_select": ["replay.cu", "replay_common.cuh", "replay_internal.h", "mot_internal.h",
                      "ptx.cuh"],
    "replay_fmha_full": ["replay_fmha.cu", "replay_common.cuh", "replay_internal.h",
                         "mot_internal.h", "ptx.cuh"],
    # backbone translators (all kernels of bt.cu)
    "bt_ffn_fused": ["bt.cu", "bt_internal.h", "gelu.cuh", "mot_internal.h", "ptx.cuh"],
}


def _code_only(text: str) -> str:
    """Source text without comments and with runs of whitespace folded, so that an edit
    to a comment does not count as a kernel change (the sources hold no string with
    a comment marker in it)."""
    text = re.sub(r"/\*.*?\*/", " ", text, flags=re.S)
    text = re.sub(r"//[^\n]*", " ", text)
    return " ".join(text.split())


def kernel_source_sha(kernel: str) -> str:
    """Hash of the code (comments left out) of the sources a kernel is built from."""
    h = hashlib.sha256()
    csrc = os.path.join(ROOT, "paper_2607_28979_gb300", "csrc")
    for n in KERNEL_SOURCES.get(kernel, sorted(os.listdir(csrc))):
        if n.endswith((".cu", ".cuh", ".h")):
            with open(os.path.join(csrc, n), encoding="utf-8") as f:
                h.update(_code_only(f.read()).encode())
    return h.hexdigest()[:16]


def recorded_traffic(kernel: str, workload: str):
    """DRAM bytes per launch from the committed ncu summary, if it was taken on
    the current kernel sources; else None."""
    p = os.path.join(ROOT, "profiles", "dram_traffic.txt")
    if not os.path.exists(p):
        return None
    sha = kernel_source_sha(kernel)
    for line in open(p):
        f = dict(kv.split("=", 1) for kv in line.split() if "=" in kv)
        if f.get("kernel") == kernel and f.get("workload") == workload and f.get("source_sha") == sha:
            return float(f["bytes_per_launch"])
    return None


class ClockSampler:
    """nvidia-smi samples (every 200 ms) during the timed region."""
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.path = None

    def start(self):
        fd, self.path = tempfile.mkstemp(prefix="mot_clocks_", suffix=".csv")
        os.close(fd)
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.gpu), f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "200"],
                stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
        except (OSError, FileNotFoundError):
            self.proc = None
        time.sleep(0.3)

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        time.sleep(0.25)
        self.proc.terminate()
        self.proc.wait(timeout=10)
        rows = []
        for line in open(self.path):
            parts = [x.strip() for x in line.split(",")]
            if len(parts) >= 9:
                rows.append(parts)
        os.unlink(self.path)
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"]}

        def num(x):
            try:
                return float(x)
            except ValueError:
                return None
        sm = [num(r[1]) for r in rows if num(r[1]) is not None]
        smax = [num(r[2]) for r in rows if num(r[2]) is not None]
        pw = [num(r[3]) for r in rows if num(r[3]) is not None]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in rows for i in range(4) if r[5 + i].lower() == "active"})
        # samples under load: power above the midpoint of the observed range
        if pw:
            thr = (min(pw) + max(pw)) / 2
            loaded = [num(r[1]) for r in rows if num(r[3]) is not None and num(r[3]) >= thr
                      and num(r[1]) is not None]
        else:
            loaded = sm
        return {"sm_mhz": statistics.median(loaded or sm) if sm else None,
                "sm_max_mhz": max(smax) if smax else None, "reasons": reasons,
                "samples": len(rows), "power_w_max": max(pw) if pw else None}


def reduce_max(values, world: int, device):
    """Element-wise max over all ranks of a list of floats (identity on one rank)."""
    if world == 1:
        return [float(v) for v in values]
    import torch
    import torch.distributed as dist
    t = torch.tensor([float(v) for v in values], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return t.tolist()


def aggregate_throughput(tokens_per_rank: int, world: int, seconds_max: float) -> float:
    """Whole-job throughput: every rank's tokens over the slowest rank's time."""
    return world * tokens_per_rank / seconds_max


def dist_setup(gpus: int):
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world != gpus and world > 1:
        raise SystemExit(f"--gpus {gpus} but WORLD_SIZE={world}")
    return world, rank, local


def cpu_oracle_rate(wl, sk, sv, blob, budget_s: float, seed: int = 3):
    """Tokens/s of the fp64 oracle on a bounded token sample (about budget_s)."""
    import oracle
    rng = np.random.default_rng(seed)

    def sample(n):
        b = rng.integers(0, wl.batch, size=n)
        s = np.array([rng.integers(0, wl.seq_lens[i]) for i in b])
        return b.astype(np.int32), s.astype(np.int32)
    def run(tb, ts):
        if wl.is_bt:
            oracle.bt_tokens(wl, sk, sv, blob, tb, ts)
        elif wl.is_h:
            oracle.translate_h_tokens(wl, sk, blob, tb, ts)
        else:
            oracle.translate_tokens(wl, sk, sv, blob, tb, ts)
    c = omp_cores()
    tb, ts = sample(c)   # one token per thread: measures the parallel throughput
    t0 = time.perf_counter()
    run(tb, ts)
    per_tok = max((time.perf_counter() - t0) / c, 1e-6)
    n = int(max(c, min(100000, budget_s / per_tok)))
    tb, ts = sample(n)
    t0 = time.perf_counter()
    run(tb, ts)
    dt = time.perf_counter() - t0
    return n / dt, n, dt


def omp_cores() -> int:
    v = os.environ.get("OMP_NUM_THREADS")
    if v and v.isdigit():
        return int(v)
    try:
        return len(os.sched_getaffinity(0))
    except AttributeError:
        return os.cpu_count() or 1


def run_reference(args, wl):
    """The fp64 oracle as the reference arm: each step is a bounded token sample."""
    world, rank, _ = dist_setup(args.gpus)
    if rank != 0:
        return 0
    import oracle
    oracle.build()
    sk, blob = synth.gen_cache(wl, 0), synth.gen_weights(wl)
    sv = sk if wl.is_h else synth.gen_cache(wl, 1)

    def run(tb, ts):
        if wl.is_bt:
            oracle.bt_tokens(wl, sk, sv, blob, tb, ts)
        elif wl.is_h:
            oracle.translate_h_tokens(wl, sk, blob, tb, ts)
        else:
            oracle.translate_tokens(wl, sk, sv, blob, tb, ts)
    rng = np.random.default_rng(11)
    # size the per-step sample to about 2 s of CPU work
    c = omp_cores()
    tb = np.zeros(c, np.int32)
    ts = (np.arange(c) % wl.seq_lens[0]).astype(np.int32)
    t0 = time.perf_counter()
    run(tb, ts)
    per_tok = (time.perf_counter() - t0) / c
    n = int(max(c, min(4096, 2.0 / max(per_tok, 1e-6))))

    def step():
        b = rng.integers(0, wl.batch, size=n).astype(np.int32)
        s = np.array([rng.integers(0, wl.seq_lens[i]) for i in b], dtype=np.int32)
        t = time.perf_counter()
        run(b, s)
        return time.perf_counter() - t
    for _ in range(args.warmup):
        step()
    times = [step() for _ in range(args.steps)]
    total = sum(times)
    value = n * args.steps / total
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1000 * total / args.steps,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic (seeded SplitMix64/Box-Muller caches and weights)",
        "config": {"workload": workload_desc(wl), "tokens_per_step": n,
                   "sample": f"{n} random tokens of the workload per step, all "
                             f"{'window' if wl.is_bt else 'translated'} layers"},
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": omp_cores(), "kind": "oracle",
                         "sample": f"{n} tokens per step x {args.steps} steps"},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)
    return 0


# Per-launch FLOPs of each translation kernel, from the step's algorithmic split.
def _per_launch_flops(alg):
    return {"umma_fused_translate": alg["flops_gemm1"] + alg["flops_gemm2"],
            "umma2_onchip_translate": alg["flops_gemm1"] + alg["flops_gemm2"],
            "umma2_wide_translate": alg["flops_gemm1"] + alg["flops_gemm2"],
            "umma2_gemm1_gelu_gate": alg["flops_gemm1"],
            "umma2_gemm2_combine_store": alg["flops_gemm2"],
            "umma2_sparse_gemm1": alg["flops_gemm1"],
            "umma2_sparse_gemm2": alg["flops_gemm2"],
            "umma2_proj": alg["flops_proj"],
            "umma_gemm1_gelu_gate": alg["flops_gemm1"],
            "simt_gemm1_gelu_gate": alg["flops_gemm1"],
            "umma_gemm2_combine_store": alg["flops_gemm2"],
            "simt_gemm2_combine_store": alg["flops_gemm2"]}


def choose_tensor_peak(peaks, clocks):
    """The bf16 peak that applies to this run, from its own clock record: the
    burst figure when no sample showed the power cap and the SM clock under load
    stayed at its maximum (a short timed region), else the sustained figure
    (the GPU settled at its power limit). Returns (peak TFLOP/s, kind, why)."""
    burst = peaks.get("bf16_tflops", FALLBACK_PEAKS["bf16_tflops"])
    sustained = peaks.get("bf16_tflops_sustained", FALLBACK_PEAKS["bf16_tflops_sustained"])
    reasons = (clocks or {}).get("reasons") or []
    sm, smax = (clocks or {}).get("sm_mhz"), (clocks or {}).get("sm_max_mhz")
    if "sw_power_cap" in reasons:
        return sustained, "sustained", "sw_power_cap seen during the timed region"
    if sm is None or smax is None:
        return sustained, "sustained", "no clock record"
    if sm < 0.97 * smax:
        return sustained, "sustained", f"SM clock under load {sm:.0f} of {smax:.0f} MHz"
    return burst, "burst", f"SM clock under load {sm:.0f} of {smax:.0f} MHz, no power cap"


def kernel_roofline(wl, alg, kstats, steps, peaks, peak_kind, clocks):
    """Roofline of the dominant kernel (largest share of device time): its
    algorithmic work per launch over its mean CUDA-event launch time."""
    name, (n_launch, tot_ms) = max(kstats.items(), key=lambda kv: kv[1][1])
    launches_per_step = max(1, n_launch // steps)
    avg_s = tot_ms / n_launch / 1000.0
    peak_t, which, why = choose_tensor_peak(peaks, clocks)
    burst = peaks.get("bf16_tflops", FALLBACK_PEAKS["bf16_tflops"])
    sustained = peaks.get("bf16_tflops_sustained", FALLBACK_PEAKS["bf16_tflops_sustained"])
    if wl.is_bt and name in alg["per_launch"]:
        # the slower of the kernel's FLOPs at tensor peak and its bytes at HBM peak
        fl, by = alg["per_launch"][name], alg["bytes_per_launch"][name]
        t_t, t_b = fl / (peak_t * 1e12), by / (peaks["hbm_gbs"] * 1e9)
        if t_b >= t_t:
            achieved = by / avg_s / 1e9
            return {"kernel": name, "bound": "hbm", "achieved": round(achieved, 1),
                    "peak": peaks["hbm_gbs"], "unit": "GB/s",
                    "frac": round(achieved / peaks["hbm_gbs"], 4),
                    "peak_kind": f"HBM copy, {peak_kind}",
                    "traffic": recorded_traffic(name, wl.name),
                    "algorithmic_per_launch": by, "flops_per_launch": fl,
                    "avg_launch_ms": tot_ms / n_launch}
        work = fl
    else:
        plf = _per_launch_flops(alg) if not wl.is_bt else {}
        if name not in plf:
            return {"kernel": name, "bound": "hbm", "achieved": None, "peak": peaks["hbm_gbs"],
                    "unit": "GB/s", "frac": None, "traffic": None}
        work = plf[name] / launches_per_step
    achieved = work / avg_s / 1e12
    return {"kernel": name, "bound": "tensor", "achieved": round(achieved, 1),
            "peak": peak_t, "unit": "TFLOP/s", "frac": round(achieved / peak_t, 4),
            "peak_kind": f"bf16 dense {which}, {peak_kind} ({why})",
            "frac_of_burst": round(achieved / burst, 4),
            "frac_of_sustained": round(achieved / sustained, 4),
            "traffic": recorded_traffic(name, wl.name),
            "algorithmic_per_launch": work, "avg_launch_ms": tot_ms / n_launch}


def step_roofline(alg, t_step_ms, peaks, peak_kind, clocks):
    """The whole step against max(FLOPs at the tensor peak, bytes at the HBM peak),
    with the peak this run's clocks call for, and both figures."""
    peak_t, which, _ = choose_tensor_peak(peaks, clocks)
    out = {"flops": alg["flops"], "bytes": alg["bytes"]}
    for tag, p in (("", peak_t), ("_burst", peaks.get("bf16_tflops", FALLBACK_PEAKS["bf16_tflops"])),
                   ("_sustained", peaks.get("bf16_tflops_sustained",
                                            FALLBACK_PEAKS["bf16_tflops_sustained"]))):
        t_roof = max(alg["flops"] / (p * 1e12), alg["bytes"] / (peaks["hbm_gbs"] * 1e9))
        out["roofline_ms" + tag] = 1000 * t_roof
        out["frac" + tag] = round(1000 * t_roof / t_step_ms, 4)
    out["peaks"] = (f"bf16 {peak_t} TFLOP/s ({which}), HBM {peaks['hbm_gbs']} GB/s ({peak_kind})")
    return out


class _Setup:
    """One handle with its weights and device inputs/outputs for a workload."""

    def __init__(self, M, torch, wl, args):
        self.wl = wl
        self.sk_h, self.blob = synth.gen_cache(wl, 0), synth.gen_weights(wl)
        self.sv_h = self.sk_h if wl.is_h else synth.gen_cache(wl, 1)   # MoT-h: one activation
        if wl.is_bt:
            self.h = M.mot_create_bt(*M.bt_config_from(wl))
        elif wl.is_h:
            self.h = M.mot_create_h(M.h_config_from(wl))
        else:
            self.h = M.mot_create(M.config_from(wl))
        M.mot_load_weights(self.h, self.blob)
        self.path = M.mot_get_path(self.h)
        names = {0: "split", 1: "fused", 2: "pair", 3: "onchip", 4: "wide"}
        if args.schedule != "auto" and not wl.is_bt:
            M.mot_set_schedule(self.h, {v: k for k, v in names.items()}[args.schedule])
        sched = names[M.mot_get_schedule(self.h)]
        if M.mot_get_routing(self.h) == M.ROUTING_SPARSE:
            sched = "routed (Top-K token buckets)"
        if wl.is_bt:
            sched = ("backbone scan on Top-1 token buckets (8 launches per window slot)"
                     if M.mot_get_routing(self.h) == 1 else
                     "backbone scan (7 launches per window slot)")
        self.schedule = sched
        self.bf = wl.dtype == "bf16"
        tdt = torch.bfloat16 if self.bf else torch.float32

        def dev(a):
            t = torch.from_numpy(a.view(np.int16) if self.bf else a).cuda()
            return t.view(torch.bfloat16) if self.bf else t
        self.sk, self.sv = dev(self.sk_h), dev(self.sv_h)
        self.dk = torch.zeros(wl.dst_shape(), dtype=tdt, device="cuda")
        self.dv = torch.zeros(wl.dst_shape(), dtype=tdt, device="cuda")
        self.lens = torch.tensor(wl.seq_lens, dtype=torch.int32, device="cuda")
        self.stream = torch.cuda.Stream()
        self.M = M

    def step(self):
        M, wl, B = self.M, self.wl, self.wl.batch
        if wl.is_bt:
            M.mot_translate_bt(self.h, self.sk, self.sv, self.lens, B, self.dk, self.dv, self.stream)
        elif wl.is_h:
            M.mot_translate_h(self.h, self.sk, self.lens, B, self.dk, self.dv, self.stream)
        else:
            M.mot_translate(self.h, self.sk, self.sv, self.lens, B, self.dk, self.dv, self.stream)


def time_device(M, torch, S, args, world, rank, local):
    """W warm-up steps, then K timed steps between barriers and synchronisations,
    CUDA events on the launching stream, per-kernel events and nvidia-smi clocks
    sampled during the timed region. Returns (ms per step, kernel stats, launches,
    clocks)."""
    import torch.distributed as dist
    with torch.cuda.stream(S.stream):
        for _ in range(args.warmup):
            S.step()
    S.stream.synchronize()
    if M.mot_get_device_status(S.h, S.stream) != M.MOT_OK:
        raise SystemExit(f"{S.wl.name}: device status not OK after warm-up")
    sampler = ClockSampler(local) if rank == 0 else None
    if sampler:
        sampler.start()
    M.mot_profile_enable(S.h, True)
    M.mot_profile_read(S.h)
    launches0 = M.mot_get_launch_count(S.h)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    e0.record(S.stream)
    for _ in range(args.steps):
        S.step()
    e1.record(S.stream)
    torch.cuda.synchronize()
    if world > 1:
        dist.barrier()
    elapsed_ms = e0.elapsed_time(e1)
    launches = M.mot_get_launch_count(S.h) - launches0
    kstats = M.mot_profile_read(S.h)
    M.mot_profile_enable(S.h, False)
    clocks = sampler.stop() if sampler else None
    status = M.mot_get_device_status(S.h, S.stream)
    if status != M.MOT_OK:
        raise SystemExit(f"{S.wl.name}: device status {M.mot_status_string(status)}")
    return elapsed_ms / args.steps, kstats, launches, clocks


# The bf16 model pairs reported beside the headline workload in one line.
PER_CONFIG = ["gpt2s_opt125m", "qwen05_qwen15", "gpt2m_qwen7"]


def run_mot(args, wl):
    world, rank, local = dist_setup(args.gpus)
    import torch
    import torch.distributed as dist
    torch.cuda.set_device(local)
    if world > 1:
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    from paper_2607_28979_gb300 import build as mot_build
    if rank == 0 or world == 1:
        mot_build.build()
    if world > 1:
        dist.barrier()
    import paper_2607_28979_gb300.mot as M

    S = _Setup(M, torch, wl, args)
    h, sk, sv, dk, dv, lens, stream = S.h, S.sk, S.sv, S.dk, S.dv, S.lens, S.stream
    sk_h, sv_h, blob, bf, B = S.sk_h, S.sv_h, S.blob, S.bf, wl.batch
    t_step, kstats, launches, clocks = time_device(M, torch, S, args, world, rank, local)

    # ---- end to end through the host-buffer entry point (pinned memory)
    hk = torch.from_numpy(sk_h.view(np.int16) if bf else sk_h).pin_memory()
    hv = torch.from_numpy(sv_h.view(np.int16) if bf else sv_h).pin_memory()
    odt = torch.int16 if bf else torch.float32
    ok = torch.empty(wl.dst_shape(), dtype=odt).pin_memory()
    ov = torch.empty(wl.dst_shape(), dtype=odt).pin_memory()
    lens_h = np.asarray(wl.seq_lens, dtype=np.int32)
    e2e_steps = max(3, min(args.steps, 50))
    es = wl.esize
    tl = len(wl.translated_layers())

    lmap = M.mot_get_layer_map(h)
    if wl.is_bt:
        win = wl.bt_window
        bt_src = sorted({lmap[t] for t in win})

    def e2e_step():
        if wl.is_bt:   # the window's source layers in, its target layers out, on one stream
            with torch.cuda.stream(stream):
                for l in bt_src:
                    sk[l].view(torch.int16).copy_(hk[l], non_blocking=True)
                    sv[l].view(torch.int16).copy_(hv[l], non_blocking=True)
                M.mot_translate_bt(h, sk, sv, lens, B, dk, dv, stream)
                ok[win[0]:win[-1] + 1].copy_(dk[win[0]:win[-1] + 1].view(torch.int16),
                                             non_blocking=True)
                ov[win[0]:win[-1] + 1].copy_(dv[win[0]:win[-1] + 1].view(torch.int16),
                                             non_blocking=True)
        elif wl.is_h:   # device entry point with the copies around it, on the same stream
            with torch.cuda.stream(stream):
                sk.view(torch.int16).copy_(hk, non_blocking=True)
                M.mot_translate_h(h, sk, lens, B, dk, dv, stream)
                ok.copy_(dk.view(torch.int16), non_blocking=True)
                ov.copy_(dv.view(torch.int16), non_blocking=True)
        else:
            M.mot_translate_host(h, hk, hv, lens_h, B, ok, ov, stream)
    for _ in range(2):
        e2e_step()
    stream.synchronize()
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    for _ in range(e2e_steps):
        e2e_step()
    stream.synchronize()
    e2e_s = time.perf_counter() - t0
    if wl.is_bt:
        h2d = 2 * len(bt_src) * hk[0].numel() * es
        d2h = 2 * len(win) * ok[0].numel() * es
        e2e_api = "mot_translate_bt with pinned host copies of the window's layers on its stream"
    elif wl.is_h:
        h2d = hk.numel() * es
        d2h = 2 * ok.numel() * es
        e2e_api = "mot_translate_h with pinned host copies on its stream"
    else:
        used_src = len({s for s in M.mot_get_layer_map(h) if s >= 0})   # source layers copied
        h2d = 2 * used_src * wl.tokens * wl.d_src * es + 4 * B
        d2h = 2 * tl * wl.tokens * wl.d_tgt * es
        e2e_api = "mot_translate_host (pinned host buffers)"

    # ---- the host link alone: the same byte counts, pinned host -> device and
    # device -> pinned host at once on two streams (no translation)
    link_ms = _host_link_ms(torch, hk, hv, ok, ov, sk, sv, dk, dv, h2d, d2h, reps=3)

    # ---- aggregate over ranks: max time
    t_step, e2e_s = reduce_max([t_step, e2e_s], world, "cuda")
    tokens = wl.tokens
    value = aggregate_throughput(tokens, world, t_step / 1000.0)
    e2e_value = aggregate_throughput(tokens * e2e_steps, world, e2e_s)
    e2e_ms = 1000 * e2e_s / e2e_steps

    alg = algorithmic(wl, M.mot_get_layer_map(h))
    peaks, peak_kind = load_peaks()
    roof = kernel_roofline(wl, alg, kstats, args.steps, peaks, peak_kind, clocks) if rank == 0 else None
    path_str = ("tcgen05 " + S.schedule) if S.path == 1 else "simt"
    M.mot_destroy(h)
    del S, sk, sv, dk, dv, hk, hv, ok, ov
    torch.cuda.empty_cache()

    # ---- the other bf16 model pairs, device-resident, in the same run
    per_config = None
    if args.per_config:
        per_config = {}
        for name in PER_CONFIG:
            if name == wl.name:
                continue
            w2 = synth.WORKLOADS[name]
            S2 = _Setup(M, torch, w2, args)
            t2, k2, l2, c2 = time_device(M, torch, S2, args, world, rank, local)
            t2 = reduce_max([t2], world, "cuda")[0]
            if rank == 0:
                a2 = algorithmic(w2, M.mot_get_layer_map(S2.h))
                r2 = kernel_roofline(w2, a2, k2, args.steps, peaks, peak_kind, c2)
                sr = step_roofline(a2, t2, peaks, peak_kind, c2)
                per_config[name] = {
                    "workload": workload_desc(w2), "ms_per_step": t2,
                    "tokens_per_s": aggregate_throughput(w2.tokens, world, t2 / 1000.0),
                    "path": ("tcgen05 " + S2.schedule) if S2.path == 1 else "simt",
                    "step_roofline": sr,
                    "dominant_kernel": {k: r2.get(k) for k in
                                        ("kernel", "achieved", "unit", "peak", "frac",
                                         "frac_of_burst", "frac_of_sustained",
                                         "avg_launch_ms")},
                    "kernels": {k: {"launches": v[0], "total_ms": round(v[1], 3)}
                                for k, v in k2.items()},
                    "gpu_launches": l2, "clocks": c2}
            M.mot_destroy(S2.h)
            del S2
            torch.cuda.empty_cache()

    if rank == 0:
        cpu = None
        if world == 1 and not args.no_cpu_baseline:
            rate, n, dt = cpu_oracle_rate(wl, sk_h, sv_h, blob, budget_s=15.0)
            layers = (f"{wl.bt[1]} window" if wl.is_bt else f"{tl} translated")
            cpu = {"value": rate, "unit": UNIT, "cores": omp_cores(), "kind": "oracle",
                   "sample": f"{n} random tokens x all {layers} layers, {dt:.1f} s"}
        line = {
            "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": t_step, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": wl.dtype,
            "data": "synthetic (seeded SplitMix64/Box-Muller caches, N(0,1/fan_in) weights)",
            "config": {"workload": workload_desc(wl), "tokens_per_step": tokens,
                       "parallelism": "replicas" if world > 1 else "single GPU",
                       "path": path_str,
                       "l2": ("inputs larger than L2 (%.2f GB read+written per step)" % (alg["bytes"] / 1e9)
                              if not wl.is_bt else
                              "each step moves more than L2: %.2f GB of caches and weights plus "
                              "the row workspace (GBs)" % (alg["bytes"] / 1e9))},
            "roofline": roof,
            "step_roofline": step_roofline(alg, t_step, peaks, peak_kind, clocks),
            "kernels": {k: {"launches": v[0], "total_ms": round(v[1], 3),
                            "share": round(v[1] / sum(x[1] for x in kstats.values()), 4)}
                        for k, v in kstats.items()},
            "per_config": per_config,
            "cpu_baseline": cpu,
            "e2e": {"value": e2e_value, "unit": UNIT, "h2d_bytes_per_step": h2d,
                    "d2h_bytes_per_step": d2h, "steps": e2e_steps, "api": e2e_api,
                    "ms_per_step": e2e_ms,
                    "host_link_gbs": round((h2d + d2h) / (e2e_ms / 1000) / 1e9, 1),
                    "link_only_ms": link_ms,
                    "link_only_gbs": round((h2d + d2h) / (link_ms / 1000) / 1e9, 1),
                    "device_ms": t_step,
                    "overlap": round(max(link_ms, t_step) / e2e_ms, 3)},
            "gpu_launches": launches,
            "clocks": clocks,
        }
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()
    return 0


def _host_link_ms(torch, hk, hv, ok, ov, sk, sv, dk, dv, h2d, d2h, reps=3):
    """Milliseconds to move h2d bytes host -> device and d2h bytes device -> host
    at once (two streams, pinned memory, flat copies): what the host link alone
    allows per step."""
    def flat(*ts):
        return [t.view(torch.int16).reshape(-1) for t in ts]
    src_h, dst_d = flat(hk, hv), flat(sk, sv)
    src_d, dst_h = flat(dk, dv), flat(ok, ov)

    def plan(total_bytes, srcs, dsts):
        out, left = [], total_bytes // 2
        for s, d in zip(srcs, dsts):
            n = min(left, s.numel(), d.numel())
            if n > 0:
                out.append((s[:n], d[:n]))
            left -= n
        return out
    up, down = plan(h2d, src_h, dst_d), plan(d2h, src_d, dst_h)
    s1, s2 = torch.cuda.Stream(), torch.cuda.Stream()

    def once():
        with torch.cuda.stream(s1):
            for a, b in up:
                b.copy_(a, non_blocking=True)
        with torch.cuda.stream(s2):
            for a, b in down:
                b.copy_(a, non_blocking=True)
    once()
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    for _ in range(reps):
        once()
    torch.cuda.synchronize()
    return 1000 * (time.perf_counter() - t0) / reps


# ---------------------------------------------------------------- replay attention (App. C.4)

def replay_desc(wl) -> str:
    return (f"{wl.name}: replay attention over {wl.n_layers_tgt} target layers "
            f"({wl.q_heads} query / {wl.kv_heads} key-value heads of {wl.head_dim}), bottom "
            f"{wl.n_full} full causal, the rest Top-{wl.top_s} guided by the head-averaged "
            f"attention maps of {wl.n_layers_src} source layers (depth-ratio map), bf16, "
            f"batch {wl.batch} seq_lens {list(wl.seq_lens)}")


def replay_guide_layers(wl):
    """Source guidance layer pi(l) of each target layer (depth-ratio map)."""
    import oracle
    return oracle.depth_ratio_map(wl.n_layers_src, wl.n_layers_tgt)


def replay_algorithmic(wl):
    """FLOPs and bytes per step (one replay of every layer), and per kernel launch."""
    B, N, Hq, Hkv, d, S = wl.max_batch, wl.max_seq, wl.q_heads, wl.kv_heads, wl.head_dim, wl.top_s
    lens = wl.seq_lens
    keys_full = sum(L * (L + 1) // 2 for L in lens)
    keys_sparse = sum(sum(min(S, u + 1) for u in range(L)) for L in lens)
    fl_full = 4 * Hq * d * keys_full           # q.k and p.v, 2 FLOP each
    fl_sparse = 4 * Hq * d * keys_sparse
    T = wl.tokens
    b_qo = 2 * T * Hq * d * 2                  # queries in, outputs out
    b_kv = 2 * T * Hkv * d * 2
    b_map = sum(L * (L + 1) // 2 for L in lens) * 2   # the causal part of one guidance map
    b_sel = T * S * 4
    n_sparse = wl.n_layers_tgt - wl.n_full
    per = {
        "replay_attn_full": dict(flops=fl_full, bytes=b_qo + b_kv),
        "replay_attn_sparse": dict(flops=fl_sparse, bytes=b_qo + b_kv),
        "replay_select": dict(flops=0, bytes=b_map + b_sel),
    }
    flops = wl.n_full * fl_full + n_sparse * fl_sparse
    byts = wl.n_layers_tgt * (b_qo + b_kv) + n_sparse * b_map
    return dict(flops=flops, bytes=byts, per_launch=per)


def _replay_oracle_rate(wl, layers, budget_s, seed=5):
    """Replayed context tokens per second of the fp64 oracle: random (layer, b, h, u)
    queries for about budget_s; one token = one position through every layer and head."""
    import oracle
    rng = np.random.default_rng(seed)
    gl = replay_guide_layers(wl)

    def sample(n):
        tb = rng.integers(0, wl.batch, size=n)
        tu = (rng.random(n) * np.asarray(wl.seq_lens)[tb]).astype(np.int64)   # u < seq_len(b)
        th = rng.integers(0, wl.q_heads, size=n)
        tl = rng.integers(0, wl.n_layers_tgt, size=n)
        return tb, th, tu, tl

    def run(tb, th, tu, tl):
        for l in np.unique(tl):
            m = tl == l
            q, k, v, g = layers(int(l), gl)
            oracle.replay_tokens(wl, int(l), q, k, v, g, tb[m], th[m], tu[m])
    # calibrate on samples large enough that per-layer call overhead does not
    # dominate (doubling until one takes a second or a tenth of the budget)
    n = 4 * omp_cores()
    while True:
        smp = sample(n)
        t0 = time.perf_counter()
        run(*smp)
        dt = time.perf_counter() - t0
        if dt >= min(1.0, 0.1 * budget_s) or n >= 1 << 20:
            break
        n *= 2
    per_q = max(dt / n, 1e-8)
    n = int(max(n, min(2_000_000, budget_s / per_q)))
    smp = sample(n)
    t0 = time.perf_counter()
    run(*smp)
    dt = time.perf_counter() - t0
    per_token = wl.n_layers_tgt * wl.q_heads
    return n / dt / per_token, n, dt


def _replay_host_inputs(wl):
    """Per-layer (q, k, v) and the guidance maps of the source layers in use, bf16
    bits on the host; returns (layers(l, gl) -> (q, k, v, guide or None), maps)."""
    gl = replay_guide_layers(wl)
    used = sorted({gl[l] for l in range(wl.n_full, wl.n_layers_tgt)})
    maps = {s: synth.gen_guide(wl, s) for s in used}
    qkv = {l: synth.gen_replay_qkv(wl, l) for l in range(wl.n_layers_tgt)}

    def layers(l, g_layers):
        q, k, v = qkv[l]
        return q, k, v, (maps[g_layers[l]] if l >= wl.n_full else None)
    return layers, qkv, maps


def run_replay_reference(args, wl):
    world, rank, _ = dist_setup(args.gpus)
    if rank != 0:
        return 0
    import oracle
    oracle.build()
    layers, _, _ = _replay_host_inputs(wl)
    times, ns = [], []
    for i in range(args.warmup + args.steps):
        rate, n, dt = _replay_oracle_rate(wl, layers, budget_s=2.0, seed=100 + i)
        if i >= args.warmup:
            times.append(dt)
            ns.append(n)
    per_token = wl.n_layers_tgt * wl.q_heads
    value = sum(ns) / sum(times) / per_token
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1000 * sum(times) / args.steps,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic (seeded queries, replay caches and source guidance maps)",
        "config": {"workload": replay_desc(wl),
                   "sample": "random (layer, batch, head, position) queries, about 2 s per step; "
                             "a token = one position through every layer and head"},
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": omp_cores(), "kind": "oracle",
                         "sample": f"{sum(ns)} queries over {args.steps} steps"},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)
    return 0


def run_replay(args, wl):
    world, rank, local = dist_setup(args.gpus)
    import torch
    import torch.distributed as dist
    torch.cuda.set_device(local)
    if world > 1:
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    from paper_2607_28979_gb300 import build as mot_build
    if rank == 0 or world == 1:
        mot_build.build()
    if world > 1:
        dist.barrier()
    import paper_2607_28979_gb300.mot as M

    layers, qkv_h, maps_h = _replay_host_inputs(wl)
    gl = replay_guide_layers(wl)
    h = M.mot_create_replay(M.replay_config_from(wl))

    def dev(a):
        return torch.from_numpy(a.view(np.int16)).cuda()
    qkv = {l: tuple(dev(a) for a in qkv_h[l]) for l in qkv_h}
    maps = {s: dev(m) for s, m in maps_h.items()}
    out = torch.empty((wl.max_batch, wl.q_heads, wl.max_seq, wl.head_dim), dtype=torch.int16,
                      device="cuda")
    lens = torch.tensor(wl.seq_lens, dtype=torch.int32, device="cuda")
    stream = torch.cuda.Stream()
    B = wl.batch
    outs = {}

    def step(dst=None):
        for l in range(wl.n_layers_tgt):
            q, k, v = qkv[l]
            g = maps[gl[l]] if l >= wl.n_full else None
            M.mot_replay_attention(h, l, q, k, v, g, lens, B, out if dst is None else dst[l],
                                   stream)

    with torch.cuda.stream(stream):
        for _ in range(args.warmup):
            step()
    stream.synchronize()
    sampler = ClockSampler(local) if rank == 0 else None
    if sampler:
        sampler.start()
    M.mot_profile_enable(h, True)
    M.mot_profile_read(h)
    launches0 = M.mot_get_launch_count(h)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    e0.record(stream)
    for _ in range(args.steps):
        step()
    e1.record(stream)
    torch.cuda.synchronize()
    if world > 1:
        dist.barrier()
    elapsed_ms = e0.elapsed_time(e1)
    launches = M.mot_get_launch_count(h) - launches0
    kstats = M.mot_profile_read(h)
    M.mot_profile_enable(h, False)
    clocks = sampler.stop() if sampler else None

    # end to end: every layer's inputs copied in from pinned host memory and its
    # output copied back, on the replay stream
    pin = lambda a: torch.from_numpy(a.view(np.int16)).pin_memory()
    qkv_p = {l: tuple(pin(a) for a in qkv_h[l]) for l in qkv_h}
    maps_p = {s: pin(m) for s, m in maps_h.items()}
    out_p = torch.empty((wl.n_layers_tgt,) + tuple(out.shape), dtype=torch.int16).pin_memory()

    def e2e_step():
        with torch.cuda.stream(stream):
            for l in range(wl.n_layers_tgt):
                for dsta, srca in zip(qkv[l], qkv_p[l]):
                    dsta.copy_(srca, non_blocking=True)
                if l >= wl.n_full:
                    maps[gl[l]].copy_(maps_p[gl[l]], non_blocking=True)
                q, k, v = qkv[l]
                M.mot_replay_attention(h, l, q, k, v, maps[gl[l]] if l >= wl.n_full else None,
                                       lens, B, out, stream)
                out_p[l].copy_(out, non_blocking=True)
    e2e_step()
    stream.synchronize()
    e2e_steps = 3
    t0 = time.perf_counter()
    for _ in range(e2e_steps):
        e2e_step()
    stream.synchronize()
    e2e_s = time.perf_counter() - t0
    h2d = sum(a.numel() * 2 for l in qkv_p for a in qkv_p[l]) + \
        sum(maps_p[gl[l]].numel() * 2 for l in range(wl.n_full, wl.n_layers_tgt))
    d2h = out_p.numel() * 2

    t_step, e2e_s = reduce_max([elapsed_ms / args.steps, e2e_s], world, "cuda")
    value = aggregate_throughput(wl.tokens, world, t_step / 1000.0)
    e2e_value = aggregate_throughput(wl.tokens * e2e_steps, world, e2e_s)
    if rank == 0:
        alg = replay_algorithmic(wl)
        peaks, peak_kind = load_peaks()
        name, (n_launch, tot_ms) = max(kstats.items(), key=lambda kv: kv[1][1])
        per = alg["per_launch"].get(name)
        avg_s = tot_ms / n_launch / 1000.0
        peak_t = peaks.get("bf16_tflops_sustained", FALLBACK_PEAKS["bf16_tflops_sustained"])
        t_t, t_b = per["flops"] / (peak_t * 1e12), per["bytes"] / (peaks["hbm_gbs"] * 1e9)
        if t_t >= t_b:
            ach = per["flops"] / avg_s / 1e12
            roof = {"kernel": name, "bound": "tensor", "achieved": round(ach, 2), "peak": peak_t,
                    "unit": "TFLOP/s", "frac": round(ach / peak_t, 4),
                    "peak_kind": f"bf16 dense sustained, {peak_kind}",
                    "traffic": recorded_traffic(name, wl.name),
                    "algorithmic_per_launch": per["flops"], "avg_launch_ms": 1000 * avg_s}
        else:
            ach = per["bytes"] / avg_s / 1e9
            roof = {"kernel": name, "bound": "hbm", "achieved": round(ach, 1),
                    "peak": peaks["hbm_gbs"], "unit": "GB/s", "frac": round(ach / peaks["hbm_gbs"], 4),
                    "peak_kind": f"HBM copy, {peak_kind}", "traffic": recorded_traffic(name, wl.name),
                    "algorithmic_per_launch": per["bytes"], "avg_launch_ms": 1000 * avg_s}
        t_roof = max(alg["flops"] / (peaks["bf16_tflops"] * 1e12), alg["bytes"] / (peaks["hbm_gbs"] * 1e9))
        cpu = None
        if world == 1 and not args.no_cpu_baseline:
            rate, n, dt = _replay_oracle_rate(wl, layers, budget_s=15.0)
            cpu = {"value": rate, "unit": UNIT, "cores": omp_cores(), "kind": "oracle",
                   "sample": f"{n} random (layer, batch, head, position) queries, {dt:.1f} s; "
                             f"a token = one position through all {wl.n_layers_tgt} layers and "
                             f"{wl.q_heads} heads"}
        line = {
            "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": t_step, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
            "data": "synthetic (seeded N(0,1) queries and replay caches; guidance maps with "
                    "sink, recency and heavy-column structure)",
            "config": {"workload": replay_desc(wl), "tokens_per_step": wl.tokens,
                       "parallelism": "replicas" if world > 1 else "single GPU",
                       "l2": "each step reads %.2f GB (queries, caches, guidance maps), more than L2"
                             % (alg["bytes"] / 1e9)},
            "roofline": roof,
            "step_roofline": {"flops": alg["flops"], "bytes": alg["bytes"],
                              "roofline_ms": 1000 * t_roof, "frac": round(1000 * t_roof / t_step, 4),
                              "peaks": f"bf16 {peaks['bf16_tflops']} TFLOP/s burst, HBM {peaks['hbm_gbs']} GB/s ({peak_kind})"},
            "kernels": {k: {"launches": v[0], "total_ms": round(v[1], 3),
                            "share": round(v[1] / sum(x[1] for x in kstats.values()), 4)}
                        for k, v in kstats.items()},
            "cpu_baseline": cpu,
            "e2e": {"value": e2e_value, "unit": UNIT, "h2d_bytes_per_step": h2d,
                    "d2h_bytes_per_step": d2h, "steps": e2e_steps,
                    "api": "mot_replay_attention per layer with pinned host copies of its inputs "
                           "and output on its stream"},
            "gpu_launches": launches,
            "clocks": clocks,
        }
        print(json.dumps(line), flush=True)
    M.mot_destroy(h)
    if world > 1:
        dist.destroy_process_group()
    return 0


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=500)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=["mot", "reference"], default="mot")
    ap.add_argument("--workload", default=DEFAULT_WORKLOAD,
                    choices=sorted(synth.WORKLOADS) + sorted(synth.REPLAY_WORKLOADS))
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--per-config", dest="per_config", action="store_true", default=None,
                    help="also time the other bf16 model pairs (device-resident) in the same "
                         "run (default: on for the headline workload)")
    ap.add_argument("--no-per-config", dest="per_config", action="store_false")
    ap.add_argument("--schedule", choices=["auto", "wide", "onchip", "pair", "fused", "split"],
                    default="auto",
                    help="tcgen05 launch schedule: the library's default for the shape, the "
                         "on-chip kernel on clusters of two CTA pairs (D_t = 512), the "
                         "on-chip GEMM1-GELU-GEMM2 kernel (D_s <= 128, D_t = 256), GEMMs on CTA "
                         "pairs (2-SM MMA), one fused persistent launch, or GEMMs on single SMs")
    ap.add_argument("--top-k", type=int, default=0,
                    help="route each token to its top-k translators (0: the workload's gate); "
                         "with 0 < k < E the translators run on token buckets")
    ap.add_argument("--n-layers", type=int, default=0,
                    help="keep only the first N layers of both models (smaller profiling case)")
    ap.add_argument("--seq-div", type=int, default=1,
                    help="divide max_seq and every sequence length by this factor (smaller "
                         "profiling case)")
    args = ap.parse_args()
    if args.warmup < 3 and args.impl == "mot":
        args.warmup = 3
    if args.workload in synth.REPLAY_WORKLOADS:
        wl = synth.REPLAY_WORKLOADS[args.workload]
        return run_replay_reference(args, wl) if args.impl == "reference" else run_replay(args, wl)
    wl = synth.WORKLOADS[args.workload]
    if args.top_k > 0:
        wl = wl.replace(name=f"{wl.name}_top{args.top_k}", top_k=args.top_k)
    if args.n_layers > 0:
        wl = wl.replace(name=f"{wl.name}_L{args.n_layers}",
                        n_layers_src=min(args.n_layers, wl.n_layers_src),
                        n_layers_tgt=min(args.n_layers, wl.n_layers_tgt))
    if args.per_config is None:
        args.per_config = (args.workload == DEFAULT_WORKLOAD and args.top_k == 0
                           and args.n_layers == 0 and args.seq_div == 1)
    if args.seq_div > 1:
        wl = wl.replace(name=f"{wl.name}_S{args.seq_div}", max_seq=wl.max_seq // args.seq_div,
                        seq_lens=tuple(L // args.seq_div for L in wl.seq_lens))
    if args.impl == "reference":
        return run_reference(args, wl)
    return run_mot(args, wl)


if __name__ == "__main__":
    sys.exit(main())
