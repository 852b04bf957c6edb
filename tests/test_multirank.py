"""The N > 1 host path of bench.py on CPU: world size 2 over gloo.

bench.py runs one replica per GPU (independent batches, weak scaling); the
only collectives are the timing barrier and a MAX all-reduce of the step
time.  These tests run that host logic with two CPU ranks, and the
reference arm under torchrun, where rank 0 alone prints.
"""
import json
import os
import socket
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    sys.path.insert(0, ROOT)
    import torch
    import torch.distributed as dist
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import bench
    from paper_2010_14298_gb300 import workloads as wl
    w, r, _ = bench._dist()
    dist.barrier()
    slowest = bench.max_over_ranks(1.0 + 2.0 * r, torch.device("cpu"))
    sh = wl.resnet50_shapes()[5]
    L = wl.resnet50_layer(sh, 1, bench.rank_seed(r, 5))
    q.put((r, w, slowest, bench.rank_seed(r, 5), float(L.dH[:4, :4].sum())))
    dist.barrier()
    dist.destroy_process_group()


def test_two_ranks_take_the_slowest_time_and_distinct_batches():
    import torch.multiprocessing as mp
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    ps = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in ps:
        p.start()
    out = sorted(q.get(timeout=240) for _ in ps)
    for p in ps:
        p.join(timeout=60)
        assert p.exitcode == 0
    assert [o[0] for o in out] == [0, 1] and all(o[1] == 2 for o in out)
    assert all(o[2] == 3.0 for o in out)          # MAX over ranks
    assert out[0][3] != out[1][3]                  # independent batches ...
    assert out[0][4] != out[1][4]                  # ... with different values


def test_reference_arm_under_torchrun_prints_once():
    cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes=1", "--nproc-per-node", "2",
           "--master-addr", "127.0.0.1", "--master-port", str(_free_port()), "bench.py",
           "--impl", "reference", "--gpus", "2", "--steps", "1", "--warmup", "0"]
    r = subprocess.run(cmd, cwd=ROOT, capture_output=True, text=True, timeout=600)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [l for l in r.stdout.splitlines() if l.startswith("{")]
    assert len(lines) == 1
    rec = json.loads(lines[0])
    assert rec["impl"] == "reference" and rec["n_gpus"] == 2 and rec["value"] > 0
    assert rec["e2e"]["h2d_bytes_per_step"] == 0
    assert rec["cpu_baseline"]["cores"] >= 1 and rec["cpu_baseline"]["kind"] == "oracle"
