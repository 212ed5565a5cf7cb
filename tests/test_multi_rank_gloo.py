"""The N>1 path of bench.py on CPU: two gloo ranks (no GPU).

Units (request, KV head) are independent, so ranks shard request batches and
exchange nothing on the data path; the only collectives are the barrier around
the timed region and the max-over-ranks reduction of the elapsed time.
"""
import os
import socket

import pytest
import torch.multiprocessing as mp


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _rank_main(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world),
                      LOCAL_RANK=str(rank))
    import bench
    import torch.distributed as dist
    r, w, local = bench.dist_setup(None)
    assert (r, w, local) == (rank, world, rank) and dist.get_backend() == "gloo"
    bench.dist_barrier(w)
    elapsed = 1.0 + rank  # rank 1 is the slower one
    out[rank] = bench.dist_max(elapsed, w)
    # each rank draws a disjoint shard: its own seeds, the same per-rank work (weak scaling)
    out[world + rank] = bench.rank_seed(11, rank)
    dist.destroy_process_group()


@pytest.mark.timeout(120)
def test_two_gloo_ranks_max_time_and_disjoint_shards():
    world = 2
    mgr = mp.Manager()
    out = mgr.dict()
    mp.spawn(_rank_main, args=(world, _free_port(), out), nprocs=world, join=True)
    assert out[0] == out[1] == 2.0  # both ranks report the slowest rank's time
    assert out[2] != out[3]  # distinct per-rank inputs
