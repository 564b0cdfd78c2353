"""Replica sharding across ranks (no GPU): the image partition and the timing
reduction, the latter through a real 2-rank gloo process group on the CPU."""
import os
import socket

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

from paper_2609_13804_gb300.replicas import max_over_ranks, shard_images


def test_partition_covers_every_image_once_and_balances():
    n_vis = [576, 4096, 256, 1024, 2304, 576, 1024, 256, 3328]
    n_txt = [48, 64, 64, 64, 64, 64, 64, 64, 96]
    for world in (1, 2, 3, 4, 9, 12):
        parts = [shard_images(n_vis, n_txt, world, r) for r in range(world)]
        flat = sorted(b for p in parts for b in p)
        assert flat == list(range(len(n_vis)))
        loads = [sum(n_vis[b] + n_txt[b] for b in p) for p in parts]
        biggest = max(v + t for v, t in zip(n_vis, n_txt))
        assert max(loads) - min(loads) <= biggest
    # deterministic: every rank computes the same partition
    assert shard_images(n_vis, n_txt, 4, 2) == shard_images(list(n_vis), list(n_txt), 4, 2)
    with pytest.raises(ValueError):
        shard_images(n_vis, n_txt, 2, 2)


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, q):
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        mine = shard_images([576] * 16, [48] * 16, world, rank)
        got = max_over_ranks(10.0 + rank)
        q.put((rank, mine, got))
    finally:
        dist.destroy_process_group()


def test_two_gloo_ranks_shard_and_reduce():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    res = sorted(q.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    (r0, s0, m0), (r1, s1, m1) = res
    assert sorted(s0 + s1) == list(range(16)) and len(s0) == len(s1) == 8
    assert m0 == m1 == 11.0


def test_max_over_ranks_without_a_group_is_the_value():
    assert not dist.is_initialized()
    assert max_over_ranks(3.5) == 3.5
