"""Multi-rank timing aggregation of bench.py on CPU: two gloo ranks.

The operator runs as independent replicas (no data exchange); the only
collective is the timing reduction: elapsed = max over ranks, work = sum."""
import os
import socket

import pytest
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
    elapsed = [1.5, 2.0][rank]
    work = [10.0, 14.0][rank]
    t, w = bench.aggregate_over_ranks(elapsed, work, dist)
    out[rank] = (t, w)
    dist.barrier()
    dist.destroy_process_group()


def test_two_rank_aggregation_takes_max_time_and_total_work():
    port = _free_port()
    with mp.Manager() as m:
        out = m.dict()
        mp.spawn(_worker, args=(2, port, out), nprocs=2, join=True)
        res = dict(out)
    assert res[0] == (2.0, 24.0) and res[1] == (2.0, 24.0)


def test_single_process_aggregation_is_identity():
    import bench
    assert bench.aggregate_over_ranks(1.25, 3.0, None) == (1.25, 3.0)


def test_visible_pair_count_matches_brute_force():
    import numpy as np

    import bench
    lq, lk = [5, 3, 0, 4], [5, 7, 2, 2]
    brute = 0
    for a, b in zip(lq, lk):
        for i in range(a):
            brute += sum(1 for j in range(b) if j <= i + (b - a))
    assert bench.visible_pairs(lq, lk) == brute
    # the Llama-3-70B layer: 8 * 4096 * 4097 / 2 pairs, 4 * 128 * 64 FLOPs each
    from paper_2608_13499_gb300 import workloads as W
    assert bench.causal_flops(W.llama3_70b()) == 4 * 128 * 64 * 8 * 4096 * 4097 // 2
