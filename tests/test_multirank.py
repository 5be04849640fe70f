"""The N > 1 host logic of bench.py on CPU with gloo, world_size 2: ranks
shard the requests (disjoint batch streams, no data exchange) and the job
time is the slowest rank's."""
import os
import socket

import numpy as np
import torch.distributed as dist
import torch.multiprocessing as mp


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import bench
    from paper_2608_09225_gb300 import workloads as W
    ms = bench.max_over_ranks(10.0 + 5.0 * rank, world, dist, "cpu")
    w = W.make("wide", seed=bench.rank_seed(123, rank, 0), n_req=64)
    out[rank] = (ms, w.batch.tokens[:4096].copy(), w.secret)
    dist.barrier()
    dist.destroy_process_group()


def test_two_ranks_gloo():
    world = 2
    port = _free_port()
    with mp.Manager() as m:
        out = m.dict()
        mp.spawn(_worker, args=(world, port, out), nprocs=world, join=True)
        res = dict(out)
    assert res[0][0] == res[1][0] == 15.0                     # max over ranks
    assert not np.array_equal(res[0][1], res[1][1])           # disjoint request shards
    assert bench_rank_seeds_distinct()


def bench_rank_seeds_distinct():
    import bench
    seeds = {bench.rank_seed(7, r, i) for r in range(8) for i in range(64)}
    return len(seeds) == 8 * 64
