"""The multi-rank path on CPU (gloo, world size 2): replicas need no data exchange (per-row
activation units make sequences independent), and the bench takes the slowest rank's time and the
whole job's frames."""
import os
import socket

import numpy as np
import pytest

torch = pytest.importorskip("torch")
import torch.distributed as dist  # noqa: E402
import torch.multiprocessing as mp  # noqa: E402


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        import bench
        import oracle
        from paper_1607_04683_gb300 import inputs
        assert bench.dist_info() == (rank, world, 0)
        ms = 100.0 + 50.0 * rank  # rank 1 is the slowest
        slowest = bench.max_over_ranks(ms, world)
        rate = bench.whole_job_rate(300, slowest, world)
        # each rank runs its own sequences: the oracle on one rank's share equals the rows of a
        # single run over every rank's sequences (no exchange is needed to shard by sequence)
        wl = inputs.LstmWorkload("d", seed=3, num_layers=2, input_dim=5, hidden=6, proj=0, num_classes=4,
                                 batch=4, frames=5, w_range=0.5)
        params, x = wl.make()
        d = oracle.desc(2, 5, 6, 0, 4)
        mine = oracle.lstm_forward(d, params, x[rank * 2:(rank + 1) * 2])["y"]
        full = oracle.lstm_forward(d, params, x)["y"]
        out[rank] = (slowest, rate, bool(np.array_equal(mine, full[rank * 2:(rank + 1) * 2])))
    finally:
        dist.destroy_process_group()


def test_two_ranks_on_gloo():
    world, port = 2, _free_port()
    with mp.Manager() as mgr:
        out = mgr.dict()
        mp.spawn(_rank_main, args=(world, port, out), nprocs=world, join=True)
        res = dict(out)
    for r in range(world):
        slowest, rate, same = res[r]
        assert slowest == 150.0
        assert rate == pytest.approx(2 * 300 / 0.150)
        assert same
