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
