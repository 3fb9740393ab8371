"""The benchmark's multi-rank host logic on CPU with two gloo ranks: the slowest
rank's time is taken, every rank gets an independent layer, and the whole-job
throughput counts every rank's steps."""
import os
import socket
import sys

import pytest
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, out):
    sys.path.insert(0, ROOT)
    import torch
    import torch.distributed as dist
    import bench
    from paper_2604_18556_gb300 import configs as C
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        mx = bench.max_over_ranks(10.0 + 5.0 * rank, torch.device("cpu"))
        w = bench.rank_workload(C.WORKLOADS["llama8b_q_proj"], rank, world)
        gathered = [None] * world
        dist.all_gather_object(gathered, (w.seed, w.data_seed))
        out[rank] = (mx, gathered)
    finally:
        dist.destroy_process_group()


def test_two_gloo_ranks():
    world, port = 2, _free_port()
    with mp.Manager() as mgr:
        out = mgr.dict()
        mp.start_processes(_worker, args=(world, port, out), nprocs=world, start_method="spawn")
        res = dict(out)
    assert res[0][0] == res[1][0] == 15.0                 # max over ranks
    seeds = res[0][1]
    assert len(set(seeds)) == world                        # independent layers


def test_whole_job_throughput_and_single_rank():
    sys.path.insert(0, ROOT)
    import bench
    from paper_2604_18556_gb300 import configs as C
    assert bench.whole_job_steps_per_s(0.5, 1) == 2000.0
    assert bench.whole_job_steps_per_s(0.5, 4) == 8000.0
    w = C.WORKLOADS["llama8b_q_proj"]
    assert bench.rank_workload(w, 0, 1) is w
    import torch
    assert bench.max_over_ranks(3.5, torch.device("cpu")) == 3.5
