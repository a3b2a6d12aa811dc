"""The replica path of bench.py under torch.distributed, on CPU with gloo.

The draft-and-verify step shards by request with no collective on the data
path; bench.py only needs the max-over-ranks time and the whole-job units.
Two gloo ranks check that: each rank gets its own seeded requests, the time
is the slowest rank's and the throughput counts every rank's units.
"""
import os
import socket

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        import bench
        from paper_2607_20507_gb300 import workloads as W
        r, ws, lr = bench.dist_env()
        w = bench.replica_workload(W.WORKLOADS[2], r)
        lens = W.context_lengths(w)
        seconds = 0.5 + rank            # rank 1 is the slower one
        value, t = bench.aggregate_throughput(1000.0, seconds, ws, "cpu")
        q.put((rank, r, ws, lr, lens.tolist(), value, t))
    finally:
        dist.destroy_process_group()


@pytest.mark.timeout(120)
def test_two_gloo_ranks_weak_scaling():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    res = sorted(q.get(timeout=100) for _ in procs)
    for p in procs:
        p.join(timeout=30)
        assert p.exitcode == 0
    (r0, rr0, ws0, lr0, lens0, v0, t0), (r1, rr1, ws1, lr1, lens1, v1, t1) = res
    assert (rr0, rr1, ws0, ws1, lr0, lr1) == (0, 1, 2, 2, 0, 1)
    assert lens0 != lens1                       # each replica has its own requests
    assert t0 == t1 == pytest.approx(1.5)       # max over ranks
    assert v0 == v1 == pytest.approx(2 * 1000.0 / 1.5)


def test_single_process_needs_no_group():
    import bench
    v, t = bench.aggregate_throughput(10.0, 2.0, 1, "cpu")
    assert (v, t) == (5.0, 2.0)


def test_bench_helpers_byte_counts():
    import numpy as np
    import bench
    from paper_2607_20507_gb300 import workloads as W
    w = W.WORKLOADS[2]
    lens = np.full(w.batch, 1000)
    kv = w.batch * 1000 * 2 * w.n_kv_heads * w.head_dim * 2
    assert bench.attention_bytes(lens, w) > kv
    need, full = bench.accept_bytes(np.array([0] * w.batch), w, 0.7)
    assert need < full
    need_all, full_all = bench.accept_bytes(np.array([w.n_draft] * w.batch), w, 0.7)
    assert need_all == full_all
    assert bench.parse_clocks(["0, 1965, 2070, 900.1, 0x0, Not Active, Not Active, Not Active, Active"]) \
        == {"sm_mhz": 1965.0, "sm_max_mhz": 2070.0, "reasons": ["sw_power_cap"], "samples": 1}
