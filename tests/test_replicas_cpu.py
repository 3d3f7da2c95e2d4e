"""The N > 1 path of bench.py on CPU: two gloo ranks on 127.0.0.1.

The decode path shards only as replicas (one independent copy of the model per GPU, no
exchange on the data path), so what runs across ranks is the benchmark's plumbing: the
barrier around the timed region, the max over ranks of the step time, and the reference
arm, which runs on rank 0 alone.
"""
import json
import os
import socket
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank, world, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world),
                      LOCAL_RANK=str(rank))
    sys.path.insert(0, ROOT)
    import torch.distributed as dist

    import bench
    w, r, _ = bench.dist_setup(None)
    assert (w, r) == (world, rank) and dist.get_backend() == "gloo"
    bench.barrier(w)
    q.put((rank, bench.max_over_ranks(w, 1.5 + rank)))  # each rank reports its own step time
    dist.destroy_process_group()


def test_max_over_ranks_and_barrier_gloo():
    torch = pytest.importorskip("torch")
    if torch.cuda.is_available():
        pytest.skip("CPU test of the gloo path")
    import torch.multiprocessing as mp
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(120)
        assert p.exitcode == 0
    got = sorted(q.get(timeout=10) for _ in range(2))
    assert got == [(0, 2.5), (1, 2.5)]  # both ranks see the slowest rank's time


def test_reference_arm_under_torchrun_prints_once():
    torch = pytest.importorskip("torch")
    if torch.cuda.is_available():
        pytest.skip("CPU test of the gloo path")
    cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes=1", "--nproc-per-node", "2",
           "--master-addr", "127.0.0.1", "--master-port", str(_free_port()), os.path.join(ROOT, "bench.py"),
           "--impl", "reference", "--gpus", "2", "--config", "1", "--steps", "2", "--warmup", "1"]
    out = subprocess.run(cmd, capture_output=True, text=True, timeout=300, cwd=ROOT)
    assert out.returncode == 0, out.stderr[-2000:]
    lines = [json.loads(l) for l in out.stdout.splitlines() if l.startswith("{")]
    assert len(lines) == 1  # rank 0 alone runs and prints
    line = lines[0]
    assert line["impl"] == "reference" and line["n_gpus"] == 2 and line["steps"] == 2
    assert line["e2e"]["h2d_bytes_per_step"] == 0 and line["cpu_baseline"]["kind"] == "oracle"


def test_timing_block_bounds():
    # the timed steps are cut into at most five consecutive, non-empty blocks covering all K
    sys.path.insert(0, ROOT)
    import bench
    for K in range(1, 300):
        b = bench.block_bounds(K)
        assert b[0] == 0 and b[-1] == K and len(b) == min(5, K) + 1
        assert all(b[i + 1] > b[i] for i in range(len(b) - 1))
