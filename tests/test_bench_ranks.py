"""bench.py's replica path on CPU: two gloo ranks combine their timings.

With N GPUs the benchmark runs N independent replicas (the decode step has
no exchange between sequences); the job's throughput is every rank's
committed tokens over the slowest rank's time.  This runs that combination
with world_size 2 on the gloo backend, without a GPU.
"""
import os
import socket

import torch.multiprocessing as mp


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _rank(rank, port, out):
    import sys
    import torch.distributed as dist
    sys.path.insert(0, os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
    import bench
    dist.init_process_group("gloo", init_method=f"tcp://127.0.0.1:{port}", rank=rank, world_size=2)
    ms, committed = [(10.0, 100), (25.0, 60)][rank]
    dist.barrier()
    out.put((rank, bench.combine_ranks(ms, committed, 2)))
    dist.destroy_process_group()


def test_two_replicas_take_max_time_and_sum_tokens():
    ctx = mp.get_context("spawn")
    out = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank, args=(r, port, out)) for r in range(2)]
    for p in procs:
        p.start()
    res = dict(out.get(timeout=120) for _ in range(2))
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    assert res[0] == res[1] == (25.0, 160.0)


def test_single_rank_is_identity():
    import sys
    sys.path.insert(0, os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
    import bench
    assert bench.combine_ranks(12.5, 7, 1) == (12.5, 7.0)
