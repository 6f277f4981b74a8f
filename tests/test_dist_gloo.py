"""The multi-rank bench path on CPU: two gloo ranks, the barrier and the
max-over-ranks timing that bench.py uses when launched with N > 1 replicas."""
import os
import socket

import torch
import torch.distributed as dist
import torch.multiprocessing as mp


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, out):
    os.environ["CUDA_VISIBLE_DEVICES"] = ""  # CPU ranks (gloo) even on a GPU machine
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world),
                      LOCAL_RANK=str(rank))
    import bench
    w, r, _ = bench.dist_setup(None)
    assert (w, r) == (world, rank)
    bench.barrier(w)
    t = bench.max_over_ranks(10.0 + 5.0 * rank, w)   # each rank's own timing
    out[rank] = t
    dist.destroy_process_group()


def test_two_replicas_share_the_max_time():
    port = _free_port()
    out = mp.Manager().dict()
    mp.spawn(_worker, args=(2, port, out), nprocs=2, join=True)
    assert out[0] == 15.0 and out[1] == 15.0


def test_single_rank_is_identity():
    import bench
    assert bench.max_over_ranks(3.5, 1) == 3.5
    assert bench.dist_setup(None)[0] == int(os.environ.get("WORLD_SIZE", "1"))
    torch.zeros(1)
