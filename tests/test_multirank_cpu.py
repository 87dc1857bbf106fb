"""The N > 1 benchmark path on CPU: two gloo ranks (replicas, no data-path
collective). The max-over-ranks timing, the whole-job throughput and the
reference arm's rank handling are the host logic that runs under torchrun."""
import os
import socket
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
torch = pytest.importorskip("torch")
import torch.distributed as dist          # noqa: E402
import torch.multiprocessing as mp        # noqa: E402


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, out):
    sys.path.insert(0, ROOT)
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import bench
    # each replica timed its own steps; rank 1 was slower
    mine = [2.0 + rank, 10.0 - rank]
    got = bench.reduce_max(mine, world, "cpu")
    dist.barrier()
    out.put((rank, got, bench.aggregate_throughput(8192, world, got[0] / 1000.0)))
    dist.destroy_process_group()


def test_two_gloo_ranks_take_the_max_over_ranks():
    world, port = 2, _free_port()
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    procs = [ctx.Process(target=_rank_main, args=(r, world, port, q)) for r in range(world)]
    for p in procs:
        p.start()
    res = dict((r, (g, v)) for r, g, v in (q.get(timeout=120) for _ in range(world)))
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    for r in range(world):
        assert res[r][0] == [3.0, 10.0]              # slowest rank per quantity
        assert res[r][1] == pytest.approx(2 * 8192 / 3e-3)


def test_single_rank_is_identity():
    sys.path.insert(0, ROOT)
    import bench
    assert bench.reduce_max([1.5, 2.5], 1, "cpu") == [1.5, 2.5]
    assert bench.aggregate_throughput(100, 1, 0.5) == 200


def test_reference_arm_other_ranks_exit_without_work(monkeypatch):
    sys.path.insert(0, ROOT)
    import bench
    import synth

    class Args:
        gpus, steps, warmup = 2, 1, 0
    monkeypatch.setenv("WORLD_SIZE", "2")
    monkeypatch.setenv("RANK", "1")
    monkeypatch.setenv("LOCAL_RANK", "1")
    called = []
    monkeypatch.setattr(synth, "gen_cache", lambda *a, **k: called.append(1))
    assert bench.run_reference(Args(), synth.WORKLOADS["tiny_fp32"]) == 0
    assert called == []
