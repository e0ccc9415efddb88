"""The multi-rank path of bench.py on CPU: two gloo ranks (replicas, weak scaling).  Every rank
decodes its own share of the users, nothing is exchanged on the data path, and the job's time is the
slowest rank's."""
import os
import socket

import numpy as np
import pytest
import torch.multiprocessing as mp


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank, world, port, out):
    import torch.distributed as dist
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import bench
    import synth
    w = synth.workload("tiny")
    users = 3
    all_prompts = synth.make_prompts(users * world, w.prompt_len, w.target.vocab, w.seed)
    mine = bench.shard_users(all_prompts, rank, world)
    ms_local = 100.0 + 50.0 * rank   # rank 1 is the slow one
    ms = bench.job_ms(ms_local, world)
    rate = bench.job_rate(len(mine), world, 4, ms)
    out[rank] = (len(mine), [int(p[0]) for p in mine], ms, rate)
    dist.barrier()
    dist.destroy_process_group()


def test_two_gloo_ranks_shard_users_and_take_the_slowest_time():
    world = 2
    port = _free_port()
    with mp.Manager() as mgr:
        out = mgr.dict()
        mp.start_processes(_rank, args=(world, port, out), nprocs=world, start_method="spawn")
        res = dict(out)
    import synth
    w = synth.workload("tiny")
    all_prompts = synth.make_prompts(3 * world, w.prompt_len, w.target.vocab, w.seed)
    firsts = res[0][1] + res[1][1]
    assert firsts == [int(p[0]) for p in all_prompts]          # disjoint shares covering every user
    assert res[0][0] == res[1][0] == 3
    assert res[0][2] == res[1][2] == 150.0                     # max over ranks
    assert res[0][3] == pytest.approx(3 * 2 * 4 / 0.150)       # whole-job lists / s
