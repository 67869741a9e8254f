"""The N > 1 host logic of bench.py on CPU ranks (gloo, world size 2).

bench.py under torchrun runs one replica per rank: a barrier and a max over
ranks around the timed region, and a single JSON line from rank 0.  These
tests run that logic with two CPU processes: the helpers directly, and the
reference arm (the oracle, which needs no GPU) through torch.distributed.run.
"""
import json
import os
import socket
import subprocess
import sys

import pytest
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, out):
    os.environ.update({"MASTER_ADDR": "127.0.0.1", "MASTER_PORT": str(port), "WORLD_SIZE": str(world),
                       "RANK": str(rank), "LOCAL_RANK": str(rank)})
    sys.path.insert(0, ROOT)
    import argparse

    import bench

    w, r, local = bench.dist_init(argparse.Namespace(impl="reference"))
    assert (w, r, local) == (world, rank, rank)
    bench.barrier(w)
    # each rank reports a different time; every rank must see the slowest
    got = bench.allreduce_max(1.5 + rank, w, "cpu")
    out.put((rank, got))
    import torch.distributed as dist

    dist.destroy_process_group()


def test_barrier_and_max_over_ranks():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(120)
        assert p.exitcode == 0
    got = sorted(q.get(timeout=5) for _ in range(2))
    assert got == [(0, 2.5), (1, 2.5)]


def test_reference_arm_two_ranks_prints_one_line():
    # blocksparse keeps the oracle sample small; rank 1 must exit 0 without work
    port = _free_port()
    cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes=1", "--nproc-per-node=2",
           "--master-addr=127.0.0.1", f"--master-port={port}", "bench.py", "--impl", "reference",
           "--workload", "blocksparse", "--gpus", "2", "--steps", "1", "--warmup", "0",
           "--ref-step-seconds", "0.3"]
    env = dict(os.environ, OMP_NUM_THREADS="1")
    r = subprocess.run(cmd, cwd=ROOT, env=env, capture_output=True, text=True, timeout=300)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [ln for ln in r.stdout.splitlines() if ln.startswith("{")]
    assert len(lines) == 1, r.stdout[-2000:]
    d = json.loads(lines[0])
    assert d["impl"] == "reference" and d["steps"] == 1 and d["value"] > 0
    assert d["cpu_baseline"]["kind"] == "oracle" and d["e2e"]["h2d_bytes_per_step"] == 0


if __name__ == "__main__":
    pytest.main([__file__, "-q"])
