"""The N > 1 path of bench.py on CPU: world_size-2 gloo ranks aggregate their step times (max)
and verified tokens (sum); each rank's batch is its own replica, so nothing else is exchanged."""
import os
import socket

import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, out):
    import sys
    import torch
    import torch.distributed as dist
    sys.path.insert(0, ROOT)
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import bench
    total_ms, verified = bench.aggregate_ranks(10.0 + 5.0 * rank, 100 + rank, world, torch.device("cpu"))
    out[rank] = (total_ms, verified)
    dist.destroy_process_group()


def test_two_gloo_ranks_aggregate_max_time_and_total_tokens():
    mgr = mp.get_context("spawn").Manager()
    out = mgr.dict()
    port = _free_port()
    mp.start_processes(_worker, args=(2, port, out), nprocs=2, join=True, start_method="spawn")
    assert out[0] == (15.0, 201) and out[1] == (15.0, 201)


def test_single_rank_is_identity():
    import sys
    sys.path.insert(0, ROOT)
    import bench
    assert bench.aggregate_ranks(3.5, 7, 1, None) == (3.5, 7)
