"""Multi-rank host logic on CPU with the gloo backend (world size 2): unit sharding, the barrier
and the max-over-ranks timing that bench.py uses, and the one-line output contract of
bench.py's reference arm under torchrun."""
import json
import os
import socket
import subprocess
import sys

import pytest
import torch.multiprocessing as mp

from paper_2606_10531_gb300 import dist as lcq_dist

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def test_shard_covers_every_unit_once():
    for n in (0, 1, 7, 8, 13, 152):
        for world in (1, 2, 3, 4, 8):
            seen = []
            sizes = []
            for r in range(world):
                rg = lcq_dist.shard(n, r, world)
                seen.extend(rg)
                sizes.append(len(rg))
            assert seen == list(range(n))
            assert max(sizes) - min(sizes) <= 1
    with pytest.raises(ValueError):
        lcq_dist.shard(4, 2, 2)


def _worker(rank, world, port, out):
    os.environ.update({"RANK": str(rank), "LOCAL_RANK": str(rank), "WORLD_SIZE": str(world),
                       "MASTER_ADDR": "127.0.0.1", "MASTER_PORT": str(port)})
    lcq_dist.init("gloo")
    r, _, w = lcq_dist.rank_world()
    lcq_dist.barrier()
    mx = lcq_dist.max_over_ranks(1.5 + r)       # per-rank "elapsed time"
    units = list(lcq_dist.shard(7, r, w))
    out.put((r, w, mx, units))
    lcq_dist.finalize()


def test_two_gloo_ranks_barrier_max_and_shards():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    res = sorted(q.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    assert [r[0] for r in res] == [0, 1]
    assert all(r[1] == 2 for r in res)
    assert all(r[2] == 2.5 for r in res)                 # max over ranks seen by both
    assert res[0][3] + res[1][3] == list(range(7))


def test_reference_arm_under_torchrun_prints_one_line():
    port = _free_port()
    cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes=1", "--nproc-per-node", "2",
           "--master-addr", "127.0.0.1", "--master-port", str(port), os.path.join(ROOT, "bench.py"),
           "--impl", "reference", "--gpus", "2", "--steps", "1", "--warmup", "1"]
    r = subprocess.run(cmd, capture_output=True, text=True, timeout=600, cwd=ROOT)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [ln for ln in r.stdout.splitlines() if ln.startswith("{")]
    assert len(lines) == 1
    line = json.loads(lines[0])
    assert line["impl"] == "reference" and line["n_gpus"] == 2
    for key in ("metric", "value", "unit", "cpu_baseline", "e2e"):
        assert key in line
