"""The multi-GPU arrangement on CPU: one process per rank (gloo, world size 2). Each rank
drafts its own candidates (no collective on the data path); the job's time is the max
over ranks and the value counts every rank's candidates."""
import os
import socket
import sys

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, q):
    sys.path.insert(0, ROOT)
    import bench
    from paper_2607_04461_gb300 import synth
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    n_local = 3
    cands = bench.rank_candidates(rank, n_local)
    z = synth.make_latents(synth.TINY, n_local, first=cands[0])
    ms_local = 100.0 + 50.0 * rank                # rank 1 is the slow one

    def reduce_max(x):
        t = torch.tensor([x], dtype=torch.float64)
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
        return float(t.item())
    ms, value = bench.aggregate(ms_local, n_local, world, reduce_max)
    gathered = [None] * world
    dist.all_gather_object(gathered, (cands, float(z[0, 0, 0, 0])))
    dist.barrier()
    q.put((rank, ms, value, gathered))
    dist.destroy_process_group()


def test_two_ranks_shard_candidates_and_take_the_slowest_time():
    world = 2
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, world, port, q)) for r in range(world)]
    for p in procs:
        p.start()
    out = sorted(q.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    from paper_2607_04461_gb300 import synth
    for rank, ms, value, gathered in out:
        assert ms == 150.0                                   # max over ranks
        assert value == pytest.approx(2 * 3 / 0.150)         # whole-job candidates / s
        (c0, z0), (c1, z1) = gathered
        assert c0 == [0, 1, 2] and c1 == [3, 4, 5]           # disjoint candidates
        assert z1 == float(synth.make_latents(synth.TINY, 1, first=3)[0, 0, 0, 0])
