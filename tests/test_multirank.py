"""Multi-process host logic of bench.py on CPU (gloo, world size 2).

The verification step partitions by sequence: every rank verifies its own
batch and ranks exchange nothing but the timing scalar, whose maximum over
ranks is the step time.  This checks that the ranks draw different batches and
that the max-reduction every rank sees is the maximum of the ranks' values."""
import os
import socket

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, out):
    import sys
    sys.path.insert(0, ROOT)
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import bench
    import workloads as W
    seed = bench.rank_seed("tiny", rank)
    w = W.build("tiny", seed=seed, device="cpu")
    local = 1.5 + rank                      # stand-in for this rank's step time
    out[rank] = (seed, int(w.orig_tokens[:8].sum()), bench.reduce_max(local, world))
    dist.barrier()
    dist.destroy_process_group()


def test_two_ranks_partition_and_reduce_max():
    world = 2
    port = _free_port()
    mgr = mp.get_context("spawn").Manager()
    out = mgr.dict()
    mp.start_processes(_worker, args=(world, port, out), nprocs=world, join=True,
                       start_method="spawn")
    (s0, t0, m0), (s1, t1, m1) = out[0], out[1]
    assert s0 != s1 and t0 != t1            # independent batches per rank
    assert m0 == m1 == pytest.approx(2.5)   # both see the max over ranks


def test_single_rank_reduce_is_identity():
    import sys
    sys.path.insert(0, ROOT)
    import bench
    assert bench.reduce_max(3.25, 1) == 3.25
    assert bench.rank_seed("7b", 0) == 1235 and bench.rank_seed("7b", 1) == 2235
