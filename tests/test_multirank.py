"""The multi-rank path of bench.py on CPU (gloo, world size 2): each rank
streams its own video (independent units, no data-path collective); the
timed region's end is a barrier and the reported time is the max over ranks."""
import os
import socket

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _worker(rank, world, port, out):
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        import bench
        bench.barrier(world)
        t = bench.reduce_max(1.5 + rank, world)  # rank 1 is the slowest
        # each rank draws its own video: same shapes, different values
        w = bench.WL.custom("mr", batch=1, heads=2, head_dim=64,
                            tokens_per_frame=4, frames_per_chunk=2,
                            num_chunks=2, seed=5)
        q0 = bench.host_chunks(w, seed_offset=rank)[0][0]
        gathered = [torch.zeros_like(q0.float()) for _ in range(world)]
        dist.all_gather(gathered, q0.float())
        out[rank] = (t, bool(torch.equal(gathered[0], gathered[1])))
    finally:
        dist.destroy_process_group()


def test_two_ranks_take_the_max_time_and_distinct_videos():
    world = 2
    port = _free_port()
    mgr = mp.Manager()
    out = mgr.dict()
    mp.spawn(_worker, args=(world, port, out), nprocs=world, join=True)
    assert out[0][0] == out[1][0] == 2.5
    assert out[0][1] is False and out[1][1] is False


def test_single_rank_needs_no_process_group():
    import bench
    bench.barrier(1)
    assert bench.reduce_max(3.25, 1) == 3.25
