"""The N > 1 path of the benchmark on CPU: two gloo ranks (no GPU). Ranks share no data path; they own
different batches of the same shape (weak scaling) and only meet to take the slowest rank's time."""
import os
import socket

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        import bench
        import mikv_inputs as mi
        w = mi.scaled(mi.WORKLOADS["tiny"], context=64)
        wr = bench.rank_workload(w, rank)
        k, v = mi.prefill_kv(wr, 0, "cpu", heads=[0])
        t = bench.max_over_ranks(dist, 1.5 + rank, device="cpu")
        q.put((rank, t, float(k.float().sum()), tuple(k.shape), wr.batch, wr.seed))
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
    (r0, t0, s0, sh0, b0, seed0), (r1, t1, s1, sh1, b1, seed1) = res
    assert t0 == t1 == 2.5            # both ranks see the slowest rank's time
    assert sh0 == sh1 and b0 == b1    # same per-rank work
    assert seed0 != seed1 and s0 != s1  # different batches
