"""Host logic of bench.py without a GPU: the replay method's algorithmic FLOPs and
bytes against closed forms, the oracle baseline's sampling budget, and the
committed DRAM traffic records."""
import os

import numpy as np
import pytest

import bench
import synth

pytest.importorskip("torch")

# 2 batch entries of 16 and 5 positions, 4 query / 2 key-value heads of 64, S = 4,
# one full layer of 3
WL = synth.ReplayWorkload("rp_bench_tiny", 2, 3, 4, 2, 64, 2, 16, (16, 5), top_s=4, n_full=1)


def test_replay_algorithmic_closed_forms():
    a = bench.replay_algorithmic(WL)
    Hq, Hkv, d, S = 4, 2, 64, 4
    # keys per query: u + 1 on full layers, min(S, u + 1) on guided ones
    keys_full = sum(range(1, 17)) + sum(range(1, 6))                      # 136 + 15
    keys_sparse = sum(min(S, u + 1) for u in range(16)) + sum(min(S, u + 1) for u in range(5))
    assert keys_sparse == (1 + 2 + 3 + 4 * 13) + (1 + 2 + 3 + 4 + 4)
    fl_full, fl_sparse = 4 * Hq * d * keys_full, 4 * Hq * d * keys_sparse
    assert a["per_launch"]["replay_attn_full"]["flops"] == fl_full
    assert a["per_launch"]["replay_attn_sparse"]["flops"] == fl_sparse
    assert a["flops"] == 1 * fl_full + 2 * fl_sparse
    T = 21                                                                # tokens
    b_qkvo = 2 * T * Hq * d * 2 + 2 * T * Hkv * d * 2                     # q, out; k, v
    b_map = keys_full * 2                                                 # causal half of a map
    assert a["per_launch"]["replay_attn_sparse"]["bytes"] == b_qkvo
    assert a["per_launch"]["replay_select"]["bytes"] == b_map + T * S * 4
    assert a["bytes"] == 3 * b_qkvo + 2 * b_map


def test_replay_oracle_baseline_samples_for_its_budget():
    """The calibration sample must not be dominated by per-layer call overhead:
    the timed sample runs for about the budget."""
    layers = bench._replay_host_inputs(WL)[0]
    rate, n, dt = bench._replay_oracle_rate(WL, layers, budget_s=1.0)
    assert rate > 0 and n > 0
    assert 0.5 <= dt <= 3.0


def test_traffic_records_parse():
    path = os.path.join(bench.ROOT, "profiles", "dram_traffic.txt")
    recs = []
    for line in open(path):
        if line.startswith("#") or not line.strip():
            continue
        f = dict(kv.split("=", 1) for kv in line.split())
        assert set(f) >= {"kernel", "workload", "source_sha", "bytes_per_launch", "capture"}
        assert len(f["source_sha"]) == 16 and float(f["bytes_per_launch"]) > 0
        assert os.path.exists(os.path.join(bench.ROOT, "profiles", f["capture"]))
        assert f["kernel"] in bench.KERNEL_SOURCES
        recs.append(f)
    assert {r["kernel"] for r in recs} >= {"umma2_gemm1_gelu_gate", "replay_attn_sparse", "bt_ffn_fused"}
    assert bench.recorded_traffic("no_such_kernel", "gpt2s_opt125m") is None


def test_kernel_source_hash_ignores_comments_only():
    """A traffic record stays valid across comment edits, not across code edits."""
    code = "int f(int x) {\n  return x + 1;  // one more\n}\n/* note */\n"
    assert bench._code_only(code) == bench._code_only(code.replace("one more", "the successor"))
    assert bench._code_only(code) == bench._code_only(code.replace("/* note */", "/* a\nlonger note */"))
    assert bench._code_only(code) != bench._code_only(code.replace("x + 1", "x + 2"))


PEAKS = {"hbm_gbs": 6796.5, "bf16_tflops": 1928.9, "bf16_tflops_sustained": 1708.6}


def test_peak_follows_the_clock_record():
    """Burst peak only for a run that saw no power cap and kept its SM clock at max."""
    short = {"sm_mhz": 2070.0, "sm_max_mhz": 2070.0, "reasons": []}
    capped = {"sm_mhz": 1455.0, "sm_max_mhz": 2070.0, "reasons": ["sw_power_cap"]}
    low = {"sm_mhz": 1800.0, "sm_max_mhz": 2070.0, "reasons": []}
    assert bench.choose_tensor_peak(PEAKS, short)[:2] == (1928.9, "burst")
    assert bench.choose_tensor_peak(PEAKS, capped)[:2] == (1708.6, "sustained")
    assert bench.choose_tensor_peak(PEAKS, low)[:2] == (1708.6, "sustained")
    assert bench.choose_tensor_peak(PEAKS, None)[:2] == (1708.6, "sustained")


def test_kernel_and_step_roofline_recompute_from_their_own_fields():
    """frac = algorithmic work per launch / mean launch time / the named peak."""
    wl = synth.WORKLOADS["qwen7_long"]
    alg = bench.algorithmic(wl, list(range(28)))
    # GEMM1 of every (layer, X) group: E * 2 * D_s * H FLOPs per token
    assert alg["flops_gemm1"] == 56 * 61440 * 4 * 2 * 512 * 2048
    kstats = {"gate": (20, 1.0), "umma2_gemm1_gelu_gate": (280, 480.0),
              "umma2_gemm2_combine_store": (280, 360.0)}
    clocks = {"sm_mhz": 1500.0, "sm_max_mhz": 2070.0, "reasons": ["sw_power_cap"]}
    r = bench.kernel_roofline(wl, alg, kstats, 20, PEAKS, "measured", clocks)
    assert r["kernel"] == "umma2_gemm1_gelu_gate" and r["peak"] == 1708.6
    per_launch = alg["flops_gemm1"] / 14            # 280 launches over 20 steps
    assert r["algorithmic_per_launch"] == pytest.approx(per_launch)
    ach = per_launch / (480.0 / 280 / 1000) / 1e12
    assert r["achieved"] == pytest.approx(ach, abs=0.05)
    assert r["frac"] == pytest.approx(ach / 1708.6, abs=1e-4)
    assert r["frac_of_burst"] == pytest.approx(ach / 1928.9, abs=1e-4)
    s = bench.step_roofline(alg, 45.0, PEAKS, "measured", clocks)
    assert s["frac"] == pytest.approx(alg["flops"] / 1708.6e12 * 1000 / 45.0, abs=1e-4)
    assert s["frac_burst"] == pytest.approx(alg["flops"] / 1928.9e12 * 1000 / 45.0, abs=1e-4)
