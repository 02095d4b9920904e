"""The N-GPU bench path is replicas only: each rank samples independently and
the ranks meet only for the barrier and the max-over-ranks time.  Checked
with world size 2 over gloo on the CPU."""

import os
import socket

import pytest
import torch.distributed as dist
import torch.multiprocessing as mp

import bench


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    p = s.getsockname()[1]
    s.close()
    return p


def _worker(rank, world, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        mine = [10.0 + rank, 3.0 - rank]          # rank 1 is slower on the first timer
        got = bench.slowest_rank(dist, mine, "cpu")
        dist.barrier()
        q.put((rank, got, bench.job_rate(500, world, got[0] / 1e3)))
    finally:
        dist.destroy_process_group()


def test_max_over_ranks_and_whole_job_rate():
    world, port = 2, _free_port()
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    procs = [ctx.Process(target=_worker, args=(r, world, port, q)) for r in range(world)]
    for p in procs:
        p.start()
    out = [q.get(timeout=120) for _ in range(world)]
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    for rank, got, rate in out:
        assert got == [11.0, 3.0]
        assert rate == pytest.approx(500 * 2 / 0.011)


def test_single_rank_is_identity():
    assert bench.slowest_rank(None, [4.0, 5.0], "cpu") == [4.0, 5.0]
    assert bench.job_rate(50, 1, 0.1) == pytest.approx(500.0)


def test_paper_context_is_consistent():
    """The quoted speedups are the quoted latencies' ratios (Tables 1, 3, 4
    and 5), and every bf16 workload maps to its backbone's record."""
    from paper_2607_27842_gb300 import synthetic as syn
    for rec in bench.PAPER.values():
        assert len(rec["featfix_s"]) == len(rec["speedup"])
        for t, sp in zip(rec["featfix_s"], rec["speedup"]):
            assert abs(rec["vanilla_s"] / t - sp) < 0.006 * sp
    assert bench.paper_context(syn.workload("tiny")) is None
    for name, src in [("dit_xl2", "Table 5"), ("flux", "Table 1"), ("flux_512", "Table 1"), ("qwen", "Table 4"),
                      ("qwen_512", "Table 4"), ("hunyuan", "Table 3"), ("hunyuan_3f", "Table 3")]:
        rec = bench.paper_context(syn.workload(name))
        assert rec["source"] == src and rec["hardware"] == "not stated"
