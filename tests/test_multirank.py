"""The multi-rank host logic of bench.py with world size 2 on CPU (gloo):
max-over-ranks timing, whole-job throughput, and the reference arm running on
rank 0 only."""
import io
import os
import socket
import sys
from contextlib import redirect_stdout

import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, q):
    sys.path.insert(0, ROOT)
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world))
    import torch.distributed as dist
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import bench
    from paper_2608_21541_gb300 import workloads as W
    got = bench.max_over_ranks(10.0 * (rank + 1), world)
    tiny = W.Workload("C1", B=1, L=2, Hq=4, H=2, n=256, d=128, w=8, keep=(1, 8),
                      kind="planted", description="tiny")

    class Args:
        steps, warmup, seed, gpus = 2, 1, 0, world
    buf = io.StringIO()
    with redirect_stdout(buf):
        bench.run_reference(Args, tiny, rank)
    dist.barrier()
    q.put((rank, got, buf.getvalue()))
    dist.destroy_process_group()


def test_two_ranks_gloo():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    out = {}
    for _ in procs:
        rank, got, text = q.get(timeout=300)
        out[rank] = (got, text)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    assert out[0][0] == out[1][0] == 20.0
    lines0 = [ln for ln in out[0][1].splitlines() if ln.startswith("{")]
    assert len(lines0) == 1 and '"impl": "reference"' in lines0[0]
    assert out[1][1].strip() == ""


def test_job_throughput_is_weak_scaling():
    sys.path.insert(0, ROOT)
    import bench
    assert bench.job_throughput(1000, 1, 1000.0) == 1000.0
    assert bench.job_throughput(1000, 4, 1000.0) == 4000.0
