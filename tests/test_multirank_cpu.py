"""The benchmark's multi-rank path on CPU: two gloo ranks on 127.0.0.1.

Each rank of a multi-GPU run is an independent replica (there is no
exchange step in the method), so what spans ranks is only the timing
reduction (slowest rank), the throughput aggregation (units of all ranks),
the barriers, and the reference arm's rank-0-only rule."""
import json
import os
import socket
import subprocess
import sys

import pytest
import torch.multiprocessing as mp

from tests.conftest import ROOT


def free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, ms_local, units, out_q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), WORLD_SIZE=str(world),
                      RANK=str(rank), LOCAL_RANK=str(rank))
    sys.path.insert(0, ROOT)
    import bench

    class A:
        impl = "lam"
    w, r, loc = bench.dist_setup(A, backend="gloo")
    bench.barrier(w)
    ms, value = bench.aggregate_replicas(ms_local[rank], units, w)
    bench.barrier(w)
    out_q.put((r, w, loc, ms, value))
    import torch.distributed as dist
    dist.destroy_process_group()


@pytest.mark.parametrize("ms_local", [(2.0, 3.0), (5.0, 1.0)])
def test_two_gloo_ranks_take_the_slowest_rank_and_count_all_units(ms_local):
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    world, units, port = 2, 27986 * 3, free_port()
    procs = [ctx.Process(target=_rank_main, args=(r, world, port, ms_local, units, q))
             for r in range(world)]
    for p in procs:
        p.start()
    res = sorted(q.get(timeout=120) for _ in range(world))
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    slow = max(ms_local)
    for r, (rank, w, loc, ms, value) in enumerate(res):
        assert (rank, w, loc) == (r, world, r)
        assert ms == slow
        assert value == pytest.approx(units * world / (slow / 1e3))


def test_single_rank_needs_no_process_group():
    sys.path.insert(0, ROOT)
    import bench
    ms, value = bench.aggregate_replicas(4.0, 1000, 1)
    assert ms == 4.0 and value == pytest.approx(1000 / 4e-3)


def test_reference_arm_under_torchrun_prints_once_from_rank_zero():
    port = free_port()
    cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes=1", "--nproc-per-node", "2",
           "--master-addr", "127.0.0.1", "--master-port", str(port), "bench.py",
           "--impl", "reference", "--gpus", "2", "--steps", "1", "--warmup", "0"]
    env = dict(os.environ, OMP_NUM_THREADS="1")
    p = subprocess.run(cmd, cwd=ROOT, capture_output=True, text=True, timeout=600, env=env)
    assert p.returncode == 0, p.stderr[-2000:]
    lines = [l for l in p.stdout.splitlines() if l.startswith("{")]
    assert len(lines) == 1, p.stdout
    d = json.loads(lines[0])
    assert d["impl"] == "reference" and d["n_gpus"] == 2 and d["value"] > 0
    assert d["e2e"]["h2d_bytes_per_step"] == 0 and d["cpu_baseline"]["kind"] == "oracle"
