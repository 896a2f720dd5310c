"""Replica runs across ranks (host logic, CPU): the slowest rank's time and
the whole-job throughput, with two gloo ranks."""
import os
import socket

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

from paper_2606_27550_gb300 import replicas


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _worker(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world),
                      LOCAL_RANK=str(rank))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    w, r, local = replicas.dist_info()
    assert (w, r, local) == (world, rank, rank)
    # rank r "took" 10 + 5 r ms for its steps
    slow = replicas.max_over_ranks(10.0 + 5.0 * rank)
    out[rank] = slow
    dist.barrier()
    dist.destroy_process_group()


def test_max_over_ranks_two_gloo_ranks():
    world, port = 2, _free_port()
    out = mp.get_context("spawn").Manager().dict()
    mp.spawn(_worker, args=(world, port, out), nprocs=world, join=True)
    assert dict(out) == {0: 15.0, 1: 15.0}


def test_single_process_and_throughput():
    assert replicas.max_over_ranks(3.5) == 3.5  # no process group
    assert replicas.job_throughput(200, 0.5, 4) == pytest.approx(1600.0)  # weak scaling: units of all ranks
    with pytest.raises(ValueError):
        replicas.job_throughput(1, 0.0, 1)
