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


@pytest.mark.timeout(180)
def test_bench_starts_n_ranks_itself():
    """`bench.py --gpus 2` without a torch.distributed environment starts two ranks itself
    (torch.distributed.run on 127.0.0.1); every rank reports through the process group
    (gloo on a host without a GPU) and rank 0 prints them."""
    import json
    import subprocess
    import sys
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    env = {k: v for k, v in os.environ.items() if k not in ("WORLD_SIZE", "RANK", "LOCAL_RANK", "MASTER_ADDR",
                                                            "MASTER_PORT")}
    env["CUDA_VISIBLE_DEVICES"] = ""
    r = subprocess.run([sys.executable, os.path.join(root, "bench.py"), "--gpus", "2", "--launch-check"],
                       env=env, capture_output=True, text=True, timeout=170)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [json.loads(x) for x in r.stdout.splitlines() if x.startswith("{")]
    assert len(lines) == 1, r.stdout
    got = lines[0]
    assert got["world_size"] == 2 and got["ranks"] == [0, 1] and got["distinct_processes"] == 2
    assert got["backend"] == "gloo"


def test_bench_refuses_a_rank_count_that_disagrees():
    import argparse
    import bench
    os.environ.pop("WORLD_SIZE", None)
    with pytest.raises(SystemExit):
        bench.dist_setup(argparse.Namespace(gpus=2))
