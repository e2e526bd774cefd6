"""The multi-rank bookkeeping of bench.py under torch.distributed, on CPU with
the gloo backend and two ranks: rows are summed over ranks, the time is the
slowest rank's, every rank agrees on whether to repeat, and the reference arm
runs on rank 0 only."""
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
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        import bench
        rows, ms = bench.reduce_over_ranks(1000.0 * (rank + 1), 2.0 + rank, world,
                                           torch.device("cpu"))
        flag = bench.any_rank(rank == 1, world, torch.device("cpu"))
        none = bench.any_rank(False, world, torch.device("cpu"))
        ref = bench.run_reference(None, rank) if rank != 0 else "skip"
        out[rank] = (rows, ms, flag, none, ref)
    finally:
        dist.destroy_process_group()


def test_reduce_over_two_gloo_ranks():
    ctx = mp.get_context("spawn")
    with ctx.Manager() as mgr:
        out = mgr.dict()
        port = _free_port()
        procs = [ctx.Process(target=_worker, args=(r, 2, port, out)) for r in range(2)]
        for p in procs:
            p.start()
        for p in procs:
            p.join(timeout=120)
            assert p.exitcode == 0
        res = dict(out)
    for rank in range(2):
        rows, ms, flag, none, ref = res[rank]
        assert rows == 3000.0  # 1000 + 2000: units of all ranks
        assert ms == 3.0  # the slowest rank
        assert flag is True and none is False
    assert res[1][4] is None  # the reference arm prints on rank 0 only


def test_single_rank_is_identity():
    import bench
    assert bench.reduce_over_ranks(5.0, 1.5, 1, None) == (5.0, 1.5)
    assert bench.any_rank(True, 1, None) is True
