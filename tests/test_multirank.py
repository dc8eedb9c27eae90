"""The replica path of bench.py on CPU: two gloo ranks shard the candidate stream
without overlap and agree on the slowest rank's time (the only collective)."""
import os
import socket
import sys

import numpy as np
import pytest
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, q):
    sys.path.insert(0, ROOT)
    import torch.distributed as dist
    import bench
    import synth
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    B = 3
    items = bench.rank_items(rank, world, B)
    w = synth.workload("tiny", batch=B * world)
    inc, io, cand, co = synth.prompts(w, items=items)
    slowest = bench.max_over_ranks(10.0 + rank)
    q.put((rank, items, cand[co[0]:co[1]].tolist(), slowest))
    dist.barrier()
    dist.destroy_process_group()


def test_two_gloo_ranks_shard_candidates_and_share_the_max_time():
    world, port = 2, _free_port()
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    procs = [ctx.Process(target=_worker, args=(r, world, port, q)) for r in range(world)]
    for p in procs:
        p.start()
    out = sorted(q.get(timeout=120) for _ in range(world))
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    items = [set(o[1]) for o in out]
    assert items[0].isdisjoint(items[1]) and items[0] | items[1] == set(range(6))
    assert out[0][2] != out[1][2]            # different candidates per rank
    assert out[0][3] == out[1][3] == 11.0    # both ranks see the slowest rank's time


def test_single_process_max_is_identity():
    sys.path.insert(0, ROOT)
    import bench
    assert bench.max_over_ranks(3.5) == 3.5
    assert bench.rank_items(0, 1, 4) == [0, 1, 2, 3]
