"""The benchmark's multi-process path on the CPU (gloo, world size 2): the
slowest replica's time is what every rank reports, whole-job throughput
counts every replica's units, and under the torchrun launcher only rank 0
prints the (reference-arm) JSON line.  The shard path itself has no exchange
step -- replicas only -- so nothing else crosses ranks.  No GPU."""
import importlib.util
import json
import os
import socket
import subprocess
import sys

import pytest
import torch.distributed as dist
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _bench():
    spec = importlib.util.spec_from_file_location("bench_mod", os.path.join(ROOT, "bench.py"))
    m = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(m)
    return m


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank, world, port, times, out_dir):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    b = _bench()
    slowest = b.max_over_ranks(times[rank], dist, "cpu")
    value = b.replica_throughput(world, 100, slowest)
    with open(os.path.join(out_dir, "rank%d.json" % rank), "w") as f:
        json.dump({"slowest": slowest, "value": value}, f)
    dist.barrier()
    dist.destroy_process_group()


def test_slowest_replica_sets_the_time(tmp_path):
    times = [0.5, 2.0]
    mp.spawn(_rank, args=(2, _free_port(), times, str(tmp_path)), nprocs=2, join=True)
    for r in range(2):
        got = json.load(open(tmp_path / ("rank%d.json" % r)))
        assert got["slowest"] == 2.0
        assert got["value"] == pytest.approx(2 * 100 / 2.0)


def test_single_process_needs_no_group():
    b = _bench()
    assert b.max_over_ranks(1.25, None, "cpu") == 1.25
    assert b.replica_throughput(1, 50, 0.5) == 100.0


def test_reference_arm_under_torchrun_prints_one_line():
    env = dict(os.environ, REFERENCE_BUDGET_S="1")
    cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes", "1", "--nproc-per-node", "2",
           "--master-addr", "127.0.0.1", "--master-port", str(_free_port()), os.path.join(ROOT, "bench.py"),
           "--impl", "reference", "--config", "tiny", "--steps", "2", "--warmup", "1"]
    r = subprocess.run(cmd, cwd=ROOT, env=env, capture_output=True, text=True, timeout=300)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [ln for ln in r.stdout.splitlines() if ln.startswith("{")]
    assert len(lines) == 1, r.stdout
    line = json.loads(lines[0])
    assert line["impl"] == "reference" and line["value"] > 0
    assert line["cpu_baseline"]["kind"] == "oracle"
