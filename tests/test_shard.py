"""Sharding one job's (sequence, layer) pairs across ranks (bench.py --shard):
with world size 2 on CPU (gloo), each rank compresses its contiguous share
with the float64 oracle, rebases its packed offsets to the whole job, and the
gathered shares must cover every pair exactly once and reproduce the
single-rank packed cache (budgets, global offsets, kept positions, slots).
Pairs are independent (budgets never couple layers or sequences), so there is
no collective on the data path; the gather here is only the test's check."""
import os
import socket
import sys

import numpy as np
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _job():
    from paper_2608_21541_gb300 import workloads as W
    return W.Workload("C1", B=2, L=3, Hq=4, H=2, n=192, d=128, w=8, keep=(1, 6),
                      kind="planted", description="tiny sharded job")


def _compress(job, pairs):
    import oracle
    import bench
    K, V, Q = bench.draw_shard(job, pairs, 0, "cpu")
    bits = [x.contiguous().view(__import__("torch").int16).numpy().view(np.uint16)
            for x in (K, V, Q)]
    return oracle.compress(*bits, B=1, L=len(pairs), Hq=job.Hq, H=job.H, n=job.n, d=job.d,
                           w=job.w, B_live=job.B_live, threads=2)


def _worker(rank, world, port, q):
    sys.path.insert(0, ROOT)
    sys.path.insert(0, os.path.join(ROOT, "tests"))
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world))
    import torch.distributed as dist
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import bench
    job = _job()
    lo, hi = bench.shard_range(job.B * job.L, world, rank)
    pairs = bench.shard_pairs(job, world, rank)
    ref = _compress(job, pairs)
    share = dict(rank=rank, lo=lo, hi=hi, pairs=pairs, counts=ref["counts"].tolist(),
                 offsets=bench.global_offsets(ref["offsets"][:-1], lo, job.B_live),
                 positions=ref["positions"].tolist(), pk=ref["pk"].tolist())
    gathered = [None] * world
    dist.all_gather_object(gathered, share)
    if rank == 0:
        q.put(gathered)
    dist.barrier()
    dist.destroy_process_group()


def test_shard_ranges_cover_every_pair_once():
    sys.path.insert(0, ROOT)
    import bench
    for total in (1, 2, 7, 32, 80, 256):
        for world in (1, 2, 3, 4, 8):
            seen = []
            for r in range(world):
                lo, hi = bench.shard_range(total, world, r)
                assert 0 <= lo <= hi <= total
                assert hi - lo in (total // world, -(-total // world))
                seen.extend(range(lo, hi))
            assert seen == list(range(total))


def test_two_rank_shards_reproduce_the_single_rank_cache():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    shares = q.get(timeout=600)
    for p in procs:
        p.join(timeout=120)
        assert p.exitcode == 0
    sys.path.insert(0, ROOT)
    job = _job()
    full = _compress(job, [(b, l) for b in range(job.B) for l in range(job.L)])
    shares.sort(key=lambda s: s["rank"])
    pairs = [p for s in shares for p in s["pairs"]]
    assert pairs == [(b, l) for b in range(job.B) for l in range(job.L)]
    assert np.array_equal(np.concatenate([s["counts"] for s in shares]), full["counts"])
    assert np.array_equal(np.concatenate([s["offsets"] for s in shares]), full["offsets"][:-1])
    assert np.array_equal(np.concatenate([s["positions"] for s in shares]), full["positions"])
    assert np.array_equal(np.concatenate([s["pk"] for s in shares]), full["pk"])
    assert full["offsets"][-1] == job.B * job.L * job.B_live
