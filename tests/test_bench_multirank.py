"""The benchmark's multi-rank host logic on CPU with two gloo ranks: the slowest
rank's time is taken, the ranks hold disjoint shards of one layer whose loss
adds up over the ranks, and the whole job advances one layer step per step;
plus the timed-window sizing and the oracle baseline on several host cores."""
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
        sm = bench.sum_over_ranks(1.0 + rank, torch.device("cpu"))
        sh = bench.rank_shard(C.WORKLOADS["llama8b_q_proj"], rank, world)
        gathered = [None] * world
        dist.all_gather_object(gathered, (sh.rows, sh.index_offset, sh.workload.seed))
        out[rank] = (mx, sm, gathered)
    finally:
        dist.destroy_process_group()


def test_two_gloo_ranks():
    world, port = 2, _free_port()
    with mp.Manager() as mgr:
        out = mgr.dict()
        mp.start_processes(_worker, args=(world, port, out), nprocs=world, start_method="spawn")
        res = dict(out)
    assert res[0][0] == res[1][0] == 15.0                 # max over ranks
    assert res[0][1] == res[1][1] == 3.0                  # loss summed over the shards
    shards = res[0][2]
    assert [s[0] for s in shards] == [(0, 2048), (2048, 4096)]   # disjoint row blocks
    assert [s[1] for s in shards] == [0, 2048 * 4096]             # their noise offsets
    assert len({s[2] for s in shards}) == 1                       # one layer, one seed


def test_throughput_window_and_single_rank():
    sys.path.insert(0, ROOT)
    import bench
    from paper_2604_18556_gb300 import configs as C
    assert bench.layer_steps_per_s(0.5) == 2000.0
    assert bench.replays_for_window(6.8, 500.0) == 74
    assert bench.replays_for_window(900.0, 500.0) == 1
    assert bench.replays_for_window(0.0, 500.0) == 1
    w = C.WORKLOADS["llama8b_q_proj"]
    sh = bench.rank_shard(w, 0, 1)
    assert sh.workload is w and sh.index_offset == 0
    import torch
    assert bench.max_over_ranks(3.5, torch.device("cpu")) == 3.5
    # the step's algorithmic bytes (separate forward and backward + Lion passes)
    assert bench.elementwise_bytes_8d(w) == w.n * (20 * 4 + 2 + 6)
    assert bench.elementwise_bytes_8d(C.WORKLOADS["llama8b_down_proj_shift5"]) == \
        C.WORKLOADS["llama8b_down_proj_shift5"].n * (20 * 5 + 2 + 6 + 2)


def test_oracle_baseline_on_several_cores():
    """The oracle baseline spawns one single-threaded process per core on its own
    block of rows; blocks that cover the layer need no scaling."""
    sys.path.insert(0, ROOT)
    import bench
    from paper_2604_18556_gb300 import configs as C
    w = C.shrunk(C.WORKLOADS["llama8b_q_proj"], rows=24, cols=256, tokens=512)
    r = bench.time_oracle(w, cores=2, step_s=30.0, n_warm=1, n_steps=1, single=True)
    assert r["workers"] == 2 and r["rows"] == 24 and r["scale"] == 1.0
    assert r["rows_per_worker"] == 12
    assert r["full_step_s"] > 0 and r["single_core_full_step_s"] > 0
    text = bench.oracle_sample_text(w, r, 2)
    assert "whole layer" in text and "2 single-threaded" in text
    # a budget below one row's cost gives one row per worker and a scaled sample
    r = bench.time_oracle(w, cores=2, step_s=1e-9, n_warm=0, n_steps=1, single=False)
    assert r["rows_per_worker"] == 1 and r["rows"] == 2 and r["scale"] == 12.0
