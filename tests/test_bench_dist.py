"""Host logic of bench.py's multi-GPU (replica) path on CPU ranks: gloo, world size 2."""
import os
import socket
import sys

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank, ws, port, out):
    sys.path.insert(0, ROOT)
    import bench
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(ws),
                      LOCAL_RANK=str(rank))

    class Args:
        impl = "reference"  # the gloo backend: no GPU here

    got_ws, got_rank, local = bench.dist_setup(Args())
    assert (got_ws, got_rank, local) == (ws, rank, rank)
    # rank r took 10 + r ms for its frames: every rank must see the slowest, 10 + ws - 1
    t = bench.max_over_ranks(10.0 + rank, ws, "cpu")
    v = bench.job_value(ws, 4.0e9, 5, t)
    out[rank] = (t, v)
    dist.barrier()
    dist.destroy_process_group()


def test_max_over_ranks_and_job_value_two_ranks():
    ws, port = 2, _free_port()
    with mp.get_context("spawn").Manager() as m:  # no fork of this (threaded) process
        out = m.dict()
        mp.spawn(_rank, args=(ws, port, out), nprocs=ws, join=True)
        res = dict(out)
    for r in range(ws):
        t, v = res[r]
        assert t == 11.0
        # 2 ranks x 5 frames x 4 GFLOP in 11 ms
        assert v == pytest.approx(2 * 4.0e9 * 5 / 11e-3 / 1e9)


def test_single_rank_needs_no_collective():
    sys.path.insert(0, ROOT)
    import bench
    assert bench.max_over_ranks(7.5, 1, "cpu") == 7.5
    assert bench.job_value(1, 2.0e9, 10, 20.0) == pytest.approx(1000.0)
