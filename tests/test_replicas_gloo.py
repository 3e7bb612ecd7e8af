"""The N > 1 path of the bench on the host: independent replicas, one per
rank, that exchange only their timings (world size 2 over gloo on CPU)."""
import json
import os
import socket
import subprocess
import sys

import pytest

from tests.conftest import ROOT


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, results):
    import torch.distributed as dist

    sys.path.insert(0, ROOT)
    import bench

    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        # each rank's decode time; the job takes as long as the slowest rank
        mine = [12.5, 20.0][rank]
        slowest = bench.rank_max(mine, world, "cpu")
        value = bench.replica_tokens_per_s(world, 8, 100, slowest)
        results.put((rank, slowest, value))
    finally:
        dist.destroy_process_group()


def test_rank_max_and_replica_throughput_over_gloo():
    import torch.multiprocessing as mp

    world, port = 2, _free_port()
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    procs = [ctx.Process(target=_rank_main, args=(r, world, port, q)) for r in range(world)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(timeout=120)
        assert p.exitcode == 0
    got = sorted(q.get(timeout=10) for _ in range(world))
    for rank, slowest, value in got:
        assert slowest == 20.0  # the max over ranks, seen by every rank
        assert value == pytest.approx(2 * 8 * 100 / 20e-3)  # both replicas' tokens over the slowest time


def test_reference_arm_prints_once_under_torchrun():
    """Under torchrun the reference arm runs on rank 0 only; the other ranks
    exit 0 without work, so the job prints exactly one JSON line."""
    env = dict(os.environ, CUDA_VISIBLE_DEVICES="")
    cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes=1", "--nproc-per-node=2",
           "--master-addr=127.0.0.1", f"--master-port={_free_port()}", os.path.join(ROOT, "bench.py"),
           "--impl", "reference", "--config", "tiny", "--gpus", "2", "--steps", "1", "--warmup", "1"]
    r = subprocess.run(cmd, cwd=ROOT, env=env, capture_output=True, text=True, timeout=600)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [l for l in r.stdout.splitlines() if l.startswith("{")]
    assert len(lines) == 1, r.stdout[-2000:]
    d = json.loads(lines[0])
    assert d["impl"] == "reference" and d["n_gpus"] == 2 and d["value"] > 0
