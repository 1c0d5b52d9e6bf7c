"""The multi-process (replica) path of bench.py on the host, as two gloo ranks.

One process per GPU runs an independent replica of the step (there is no
exchange on the data path); the job's time is the slowest rank's timed region
and its work the sum over ranks.  These tests run that aggregation, and the
reference arm's rank handling, with world size 2 on the CPU.
"""
import io
import os
import socket
import contextlib

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

import bench


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _ranks(rank, world, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        # rank r timed (10 + r) ms and processed (100 + r) units
        t, work = bench.reduce_over_ranks(dist, torch.device("cpu"), 10.0 + rank, 100 + rank)
        # the reference arm: ranks other than 0 exit 0 without work or output
        buf = io.StringIO()
        rc = None
        if rank != 0:
            with contextlib.redirect_stdout(buf):
                rc = bench.main(["--impl", "reference", "--gpus", str(world), "--steps", "3",
                                 "--warmup", "3", "--workload", "tiny"])
        q.put((rank, t, work, rc, buf.getvalue()))
        dist.barrier()
    finally:
        dist.destroy_process_group()


def test_two_rank_replica_aggregation_and_reference_ranks():
    world, port = 2, _free_port()
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    procs = [ctx.Process(target=_ranks, args=(r, world, port, q)) for r in range(world)]
    for p in procs:
        p.start()
    res = sorted(q.get(timeout=120) for _ in range(world))
    for p in procs:
        p.join(timeout=120)
        assert p.exitcode == 0
    for rank, t, work, rc, out in res:
        assert t == 11.0                  # the slowest rank
        assert work == 201.0              # all ranks' work
        if rank != 0:
            assert rc == 0 and out == ""
