"""The multi-replica logic of bench.py on CPU: two gloo ranks (no GPU)."""
import os
import socket

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import bench
    ms = 100.0 + 50.0 * rank                       # rank 1 is the slow one
    m = bench.max_over_ranks(ms, world, device="cpu")
    v = bench.job_tokens_per_s(4096, 10, world, m)
    ids = bench.rank_batch_ids(rank, 4)
    out[rank] = (m, v, tuple(ids))
    dist.destroy_process_group()


def test_two_replicas_take_the_slowest_rank_and_count_all_tokens():
    port = _free_port()
    with mp.get_context("spawn").Manager() as mgr:
        out = mgr.dict()
        mp.spawn(_worker, args=(2, port, out), nprocs=2, join=True)
        res = dict(out)
    assert res[0][0] == res[1][0] == 150.0
    assert res[0][1] == res[1][1] == pytest.approx(4096 * 10 * 2 / 0.150)
    assert set(res[0][2]).isdisjoint(res[1][2])      # replicas train on different micro-batches
