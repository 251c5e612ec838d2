"""The N>1 host logic of bench.py on CPU: two gloo ranks (replicas only, no data-path collective).

Checks the barrier, the max-over-ranks timing reduction that bench.py applies to its timed span,
and that the reference arm prints from rank 0 only."""
import json
import os
import socket
import subprocess
import sys

import pytest
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    p = s.getsockname()[1]
    s.close()
    return p


def _worker(rank, world, port, q):
    os.environ.update(RANK=str(rank), WORLD_SIZE=str(world), LOCAL_RANK=str(rank),
                      MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    sys.path.insert(0, ROOT)
    import bench
    import torch.distributed as dist
    r, w = bench.init_dist("gloo")
    bench.barrier(w)
    got = bench.max_over_ranks(10.0 + r, w)
    q.put((r, w, got))
    dist.destroy_process_group()


def test_two_rank_barrier_and_max_reduction():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(120)
        assert p.exitcode == 0
    res = sorted(q.get(timeout=10) for _ in range(2))
    assert res == [(0, 2, 11.0), (1, 2, 11.0)]


def test_reference_arm_prints_on_rank0_only(tmp_path):
    # rank 1 of a 2-rank reference run must exit 0 without output and without work
    env = dict(os.environ, RANK="1", WORLD_SIZE="2", LOCAL_RANK="1", MASTER_ADDR="127.0.0.1",
               MASTER_PORT=str(_free_port()))
    # rank 1 alone cannot rendezvous; give it a partner that only joins the group
    port = env["MASTER_PORT"]
    code = ("import os,sys; sys.path.insert(0, %r); import bench; bench.init_dist('gloo')" % ROOT)
    env0 = dict(env, RANK="0", LOCAL_RANK="0")
    p0 = subprocess.Popen([sys.executable, "-c", code], env=env0, cwd=ROOT)
    p1 = subprocess.run([sys.executable, "bench.py", "--impl", "reference", "--steps", "1", "--warmup", "0"],
                        env=env, cwd=ROOT, capture_output=True, text=True, timeout=300)
    p0.wait(120)
    assert p1.returncode == 0, p1.stderr
    assert p1.stdout.strip() == ""
