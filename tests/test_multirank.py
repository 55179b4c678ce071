"""Host-side logic of the multi-GPU benchmark path, as gloo ranks on CPU.

Streams are independent, so ranks share no data: each rank generates its own
replicas (disjoint seeds) and the only collective is the max of the step time
over ranks."""
import os
import socket

import numpy as np
import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    p = s.getsockname()[1]
    s.close()
    return p


def _worker(rank, world, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import bench
    import synth
    ms = 10.0 + 5.0 * rank
    got = bench.max_over_ranks(ms)
    seed0 = bench.rank_seed0(rank, 8)
    spec = synth.config1(8)
    spec.seed0 = seed0
    w = synth.make_workload(spec, requests_per_stream=20)
    q.put((rank, got, seed0, w.stream_seed.tolist(), int(w.length.sum())))
    dist.barrier()
    dist.destroy_process_group()


@pytest.mark.parametrize("world", [2])
def test_ranks_time_max_and_disjoint_replicas(world):
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, world, port, q)) for r in range(world)]
    for p in procs:
        p.start()
    res = [q.get(timeout=120) for _ in range(world)]
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    res.sort()
    assert all(r[1] == 10.0 + 5.0 * (world - 1) for r in res)      # max over ranks
    seeds = [set(r[3]) for r in res]
    assert not (seeds[0] & seeds[1])                                 # disjoint replicas
    assert res[0][4] != res[1][4]


def test_single_process_max_is_identity():
    import bench
    assert bench.max_over_ranks(3.5) == 3.5
