"""The multi-replica path of bench.py on CPU: two gloo ranks.

The layer does not shard (one GPU holds every expert), so N GPUs run N
independent replicas with no collective on the data path; only the timing
uses the process group (a barrier around the timed region and the maximum
of the ranks' times). This checks that plumbing with world_size 2 on the host:
the ranks see their own RANK / WORLD_SIZE, the barrier returns, the max over
ranks is every rank's maximum, and each replica gets its own tokens with the
same weights.
"""

import os
import socket

import pytest
import torch
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, q):
    import sys

    sys.path.insert(0, ROOT)
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    torch.distributed.init_process_group("gloo", rank=rank, world_size=world)
    import bench
    from paper_2603_02376_gb300 import inputs as I

    r, w, local = bench.dist_env()
    bench.barrier(w)
    m = bench.max_over_ranks(1.5 * (rank + 1), w)
    d = bench.build_inputs(I.TINY, "cpu", rank)
    q.put((rank, r, w, local, m, float(d["x"].float().sum()), float(d["W13"].float().sum())))
    bench.barrier(w)
    torch.distributed.destroy_process_group()


def test_two_gloo_ranks_time_and_shard_like_the_bench():
    world = 2
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, world, port, q)) for r in range(world)]
    for p in procs:
        p.start()
    out = [q.get(timeout=120) for _ in range(world)]
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    out.sort()
    for rank, r, w, local, m, xs, ws in out:
        assert (r, w, local) == (rank, world, rank)
        assert m == pytest.approx(1.5 * world)          # the slowest rank sets the time
    assert out[0][5] != out[1][5]                        # own tokens per replica
    assert out[0][6] == out[1][6]                        # the same weights
