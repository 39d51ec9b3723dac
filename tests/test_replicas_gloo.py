"""The multi-GPU path of bench.py is replicas only (every rank runs the whole
workload on its own GPU; no collective on the data path).  Its host logic --
the max-over-ranks timing, the whole-job rates, and the reference arm that
only rank 0 runs -- is checked here with two gloo ranks on the CPU."""
import multiprocessing
import os
import socket
import types

import pytest


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _rank_main(rank, world, port, out):
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    import torch.distributed as dist
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        import bench
        # rank r measured 10 + r ms for the device loop and 5 - r ms end to end
        times = bench.max_over_ranks([10.0 + rank, 5.0 - rank], world)
        rates = bench.replica_rates(world, 2.0e6, 4, 10, times[0], times[1])
        args = types.SimpleNamespace(steps=1, warmup=0, batch=1, layers=1)
        ref = bench.run_reference(args, rank, world) if rank != 0 else "rank 0 runs it"
        dist.barrier()
        out.put((rank, times, rates, ref))
    finally:
        dist.destroy_process_group()


def test_replicas_two_gloo_ranks():
    world = 2
    ctx = multiprocessing.get_context("spawn")
    out = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank_main, args=(r, world, port, out)) for r in range(world)]
    for p in procs:
        p.start()
    try:
        res = sorted(out.get(timeout=120) for _ in range(world))
    finally:
        for p in procs:
            p.join(timeout=60)
            if p.is_alive():
                p.kill()
    assert [p.exitcode for p in procs] == [0, 0]
    for rank, times, rates, ref in res:
        # both ranks see the slowest replica's times
        assert times == [11.0, 5.0]
        # whole job: 2 replicas x 2 MB per step over 1.1 ms per step
        assert rates["ms_per_step"] == pytest.approx(1.1)
        assert rates["gbs"] == pytest.approx(2 * 2.0e6 / 1.1e-3 / 1e9)
        assert rates["tokens_per_s"] == pytest.approx(2 * 4 / 1.1e-3)
        assert rates["e2e_gbs"] == pytest.approx(2 * 2.0e6 / 0.5e-3 / 1e9)
    # the reference arm: rank 1 returns at once with nothing to print
    assert res[1][3] is None


def test_single_rank_needs_no_process_group():
    import bench
    assert bench.max_over_ranks([3.0, 4.0], 1) == [3.0, 4.0]
    r = bench.replica_rates(1, 1.0e9, 1, 4, 8.0, 16.0)
    assert r["ms_per_step"] == 2.0 and r["gbs"] == pytest.approx(500.0)
    assert r["e2e_gbs"] == pytest.approx(250.0)
