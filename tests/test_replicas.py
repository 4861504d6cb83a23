"""The multi-replica bench logic on CPU: two gloo ranks (the layer itself does
not shard, so `bench.py --gpus N` runs N independent replicas; the job's time
is the slowest rank's and its throughput counts every rank's tokens), and the
reference arm printing from rank 0 only."""
import json
import os
import socket
import subprocess
import sys

import pytest
import torch.distributed as dist
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)
import bench  # noqa: E402


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank, world, port, out):
    dist.init_process_group("gloo", init_method=f"tcp://127.0.0.1:{port}", rank=rank, world_size=world)
    ms = [12.5, 30.0][rank]  # rank 1 is the slow replica
    got = bench.max_over_ranks(ms, dist, "cpu")
    out[rank] = (got, bench.replica_throughput(32, 10, world, got / 1e3))
    dist.destroy_process_group()


def test_time_is_the_slowest_replica_and_tokens_count_every_rank():
    world = 2
    with mp.get_context("spawn").Manager() as m:
        out = m.dict()
        mp.spawn(_rank, args=(world, _free_port(), out), nprocs=world, join=True)
        res = dict(out)
    assert res[0][0] == res[1][0] == 30.0
    assert res[0][1] == res[1][1] == pytest.approx(32 * 10 * 2 / 0.030)


def test_single_process_needs_no_group():
    assert bench.max_over_ranks(7.0, None, "cpu") == 7.0
    assert bench.replica_throughput(32, 200, 1, 0.5) == pytest.approx(12800.0)


@pytest.mark.parametrize("rank", [0, 1])
def test_reference_arm_prints_on_rank_zero_only(rank):
    env = dict(os.environ, RANK=str(rank), WORLD_SIZE="2", LOCAL_RANK=str(rank))
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference", "--workload", "1",
                        "--steps", "1", "--warmup", "0", "--gpus", "2"],
                       cwd=ROOT, env=env, capture_output=True, text=True, timeout=300)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [l for l in r.stdout.splitlines() if l.strip()]
    if rank == 0:
        d = json.loads(lines[-1])
        assert d["impl"] == "reference" and d["n_gpus"] == 2 and d["value"] > 0
        assert d["e2e"]["h2d_bytes_per_step"] == 0
    else:
        assert lines == []
