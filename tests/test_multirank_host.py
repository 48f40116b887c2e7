"""Host logic of the multi-GPU benchmark on CPU ranks (gloo, world size 2).

Rows of different batches are independent, so N GPUs run N independent batches (weak
scaling) with no data exchange; the only collective is the timing gather, and the job time
is the slowest rank's.  Here two CPU processes stand in for the ranks."""
import os
import socket

import pytest
import torch.distributed as dist
import torch.multiprocessing as mp

import bench


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    t = 0.5 + 0.25 * rank  # rank 1 is the slow one
    times = bench.gather_times(dist, t, "cpu")
    agg = bench.aggregate(64, 100, times)
    out[rank] = (times, agg["value"], agg["seconds"], bench.rank_seed(1234, rank))
    dist.barrier()
    dist.destroy_process_group()


def test_two_rank_gather_and_aggregate():
    world, port = 2, _free_port()
    with mp.Manager() as mgr:
        out = mgr.dict()
        mp.spawn(_rank_main, args=(world, port, out), nprocs=world, join=True)
        res = dict(out)
    for rank in range(world):
        times, value, seconds, seed = res[rank]
        assert times == [0.5, 0.75]
        assert seconds == 0.75
        assert value == pytest.approx(64 * 100 * 2 / 0.75)
    assert res[0][3] != res[1][3]  # independent batches per rank


def test_aggregate_single_rank():
    agg = bench.aggregate(64, 1000, [0.065])
    assert agg["value"] == pytest.approx(64 * 1000 / 0.065) and agg["n_ranks"] == 1
