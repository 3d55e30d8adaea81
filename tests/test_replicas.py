"""Host logic of the multi-GPU benchmark (replicas only: every rank prefills its own request,
the only collective is the max of the step times), run as two gloo ranks on the CPU."""
import os
import socket

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

import bench


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank: int, world: int, port: int, q) -> None:
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        local = [812.5, 799.25][rank]
        ms = bench.max_over_ranks(local, world, torch.device("cpu"))
        q.put((rank, ms, bench.replica_tokens_per_s(124032, world, ms)))
    finally:
        dist.destroy_process_group()


def test_max_over_two_gloo_ranks():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(timeout=120)
        assert p.exitcode == 0
    got = sorted(q.get(timeout=10) for _ in range(2))
    for rank, ms, tps in got:
        assert ms == 812.5                                   # the slower replica decides
        assert tps == pytest.approx(2 * 124032 / 0.8125)     # both replicas' tokens


def test_single_rank_is_identity():
    assert bench.max_over_ranks(3.5, 1) == 3.5
    assert bench.replica_tokens_per_s(1000, 1, 500.0) == pytest.approx(2000.0)
