"""The multi-GPU path of bench.py is replicas only: one independent pool per
rank on its own trace, with no collective on the data path; the ranks meet
only to time the run (barriers, the maximum of their times) and to add up
their work.  Those host-side pieces run here as two gloo ranks on CPU."""
import os
import socket
import sys

import pytest

torch = pytest.importorskip("torch")
import torch.distributed as dist  # noqa: E402
import torch.multiprocessing as mp  # noqa: E402

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank: int, world: int, port: int, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), WORLD_SIZE=str(world), RANK=str(rank),
                      LOCAL_RANK=str(rank))
    sys.path.insert(0, ROOT)
    import bench
    ws, r, local = bench.dist_setup()
    try:
        assert (ws, r, local) == (world, rank, rank)
        assert dist.get_backend() == "gloo"
        bench.barrier(ws)
        # the job's time is the slowest rank's; its work is every rank's
        t_max = bench.max_over_ranks(ws, 1.0 + rank)
        work = bench.sum_over_ranks(ws, 100.0 * (rank + 1))
        out.put((rank, t_max, work))
    finally:
        dist.destroy_process_group()


def test_replica_timing_and_work_over_two_gloo_ranks():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank_main, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(timeout=120)
    assert all(p.exitcode == 0 for p in procs), [p.exitcode for p in procs]
    got = sorted(q.get(timeout=5) for _ in range(2))
    assert got == [(0, 2.0, 300.0), (1, 2.0, 300.0)]


def test_replica_traces_differ_by_rank():
    """Weak scaling: every rank runs the same workload shape on its own seed."""
    sys.path.insert(0, ROOT)
    from paper_2608_01657_gb300 import workloads as W
    a = W.make_workload(0, seed=1 + 0)
    b = W.make_workload(0, seed=1 + 1)
    sa, sb = next(iter(a.steps(1))), next(iter(b.steps(1)))
    assert a.spec == b.spec
    assert sa.num_requests == sb.num_requests == a.spec.requests_per_step
    assert not (sa.num_tokens == sb.num_tokens and (sa.tokens == sb.tokens).all())
