"""The multi-rank (replica) path of bench.py on CPU with gloo, world size 2: every rank
runs its own scene, the job time is the slowest rank's, the value counts every rank."""
import os
import socket

import numpy as np
import torch.multiprocessing as mp


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank, world, port, out):
    import torch.distributed as dist
    import bench
    import synth
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    ms_local = 100.0 + 50.0 * rank
    ms = bench.reduce_max_over_ranks(ms_local, world, "cpu")
    seed = bench.replica_seed(bench.WORKLOAD.seed, rank)
    tokens = synth.make_tokens(seed, 64)
    out[rank] = (ms, bench.job_value(ms, world, bench.WORKLOAD.views), seed, int(tokens.sum()))
    dist.barrier()
    dist.destroy_process_group()


def test_two_replicas_reduce_to_the_slowest_rank():
    world = 2
    port = _free_port()
    with mp.Manager() as m:
        out = m.dict()
        mp.spawn(_rank, args=(world, port, out), nprocs=world, join=True)
        res = dict(out)
    assert res[0][0] == res[1][0] == 150.0          # max over ranks
    assert np.isclose(res[0][1], 100 * 2 / 0.150)   # 100 views per rank, 2 ranks
    assert res[0][2] != res[1][2] and res[0][3] != res[1][3]  # distinct scenes
