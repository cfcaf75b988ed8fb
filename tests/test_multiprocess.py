"""The multi-process path of the benchmark (one process per GPU under torchrun) on the CPU with the
gloo backend, world size 2: the work shards with no exchange (independent requests per rank), the
only collective is the max-over-ranks step time, and the whole-job throughput counts every rank's
tokens. No GPU."""
import os
import socket

import numpy as np
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

import bench
from paper_2609_34977_gb300 import synth


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        ms = bench.max_over_ranks(3.0 + rank, dist, "cpu")  # rank 1 is the slower one
        v = synth.vision_tiles(bench.rank_seed(rank), 1, 32, 16, 2, 4)
        sums = [None] * world
        dist.all_gather_object(sums, float(v["feats"][0].sum()))
        out[rank] = (ms, bench.job_throughput(640, world, ms), sums)
    finally:
        dist.destroy_process_group()


def test_two_ranks_on_gloo():
    world = 2
    with mp.Manager() as m:
        out = m.dict()
        mp.spawn(_rank, args=(world, _free_port(), out), nprocs=world, join=True)
        res = dict(out)
    for r in range(world):
        ms, value, sums = res[r]
        assert ms == 4.0                        # every rank reports the slowest rank's time
        assert value == 640 * 2 / 0.004         # all ranks' tokens over that time
        assert sums[0] != sums[1]               # independent requests per rank


def test_single_process_needs_no_collective():
    assert bench.max_over_ranks(2.5, None, "cpu") == 2.5
    assert bench.job_throughput(640, 1, 5.0) == 128000.0
    assert bench.rank_seed(0) != bench.rank_seed(1)
    assert not np.array_equal(synth.vision_tiles(bench.rank_seed(0), 1, 8, 4, 1, 2)["feats"][0],
                              synth.vision_tiles(bench.rank_seed(1), 1, 8, 4, 1, 2)["feats"][0])
