"""The N > 1 path of bench.py on CPU: two ranks over gloo (world size 2, 127.0.0.1).  Each rank
times its own replica; the job's time is the slowest rank's, and the job's throughput counts every
rank's batch (weak scaling, no collective on the data path)."""
import os
import socket
import sys

import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank, world, port, out):
    sys.path.insert(0, ROOT)
    import torch.distributed as dist

    import bench
    dist.init_process_group("gloo", init_method=f"tcp://127.0.0.1:{port}", rank=rank, world_size=world)
    dist.barrier()
    # rank r "measured" (r + 1) ms per step and (10 - r) ms in its decode kernels
    total, dec = bench.max_over_ranks([rank + 1.0, 10.0 - rank], world, "cpu")
    out.put((rank, total, dec, bench.job_tokens_per_s(world, 16, total)))
    dist.barrier()
    dist.destroy_process_group()


def test_two_ranks_take_the_slowest_time_and_count_both_batches():
    ctx = mp.get_context("spawn")
    out = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank, args=(r, 2, port, out)) for r in range(2)]
    for p in procs:
        p.start()
    got = sorted(out.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    for rank, total, dec, tps in got:
        assert (total, dec) == (2.0, 10.0)  # the slowest rank's times, on every rank
        assert tps == 2 * 16 / 2.0e-3       # both ranks' batches over the job's step time


def test_one_rank_needs_no_process_group():
    sys.path.insert(0, ROOT)
    import bench
    assert bench.max_over_ranks([3.5, 1.0], 1, "cpu") == [3.5, 1.0]
    assert bench.job_tokens_per_s(1, 16, 8.0) == 2000.0
