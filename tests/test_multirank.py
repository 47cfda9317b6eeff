"""The multi-rank path of bench.py on CPU: world_size-2 gloo ranks, as
torchrun launches one rank per GPU.  Each rank serves its own decoding
streams (no data exchange); the ranks meet only at a barrier and the
max-over-ranks reduction of the timed region, and the whole-job value
divides every rank's work by the slowest rank's time."""
import os
import socket

import pytest
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, q):
    import sys
    sys.path.insert(0, ROOT)
    os.environ.update(RANK=str(rank), LOCAL_RANK=str(rank), WORLD_SIZE=str(world),
                      MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    import bench
    import torch.distributed as dist
    w, r, _ = bench.dist_setup()
    bench.barrier(w)
    slowest = bench.max_over_ranks(10.0 + 5.0 * r, w)
    value = bench.aggregate(w, 4, 100, slowest)
    q.put((r, w, slowest, value))
    dist.destroy_process_group()


def test_two_gloo_ranks_take_the_slowest_time():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank_main, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    got = sorted(q.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    assert [g[0] for g in got] == [0, 1]
    for _, world, slowest, value in got:
        assert world == 2 and slowest == 15.0
        # 2 ranks x 4 queries x 100 steps in 15 ms
        assert value == pytest.approx(2 * 4 * 100 / 0.015)


def test_single_rank_needs_no_process_group():
    import sys
    sys.path.insert(0, ROOT)
    import bench
    for k in ("RANK", "WORLD_SIZE", "LOCAL_RANK"):
        os.environ.pop(k, None)
    world, rank, local = bench.dist_setup()
    assert (world, rank, local) == (1, 0, 0)
    assert bench.max_over_ranks(3.5, 1) == 3.5
    assert bench.aggregate(1, 4, 2000, 2800.0) == pytest.approx(4 * 2000 / 2.8)
