"""The N > 1 path of bench.py on CPU: two gloo ranks (world size 2) run the
replica bookkeeping the GPU run uses -- rendezvous, barrier, the max over
ranks of the timed region, the whole-job rate -- and the reference arm's
non-zero ranks exit without work.  The layer itself has no cross-rank
exchange (replicas only), so no data-path collective is tested."""
import io
import multiprocessing as mp
import os
import socket
import sys
from contextlib import redirect_stdout

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank: int, world: int, port: int, q):
    os.environ.update({"MASTER_ADDR": "127.0.0.1", "MASTER_PORT": str(port), "RANK": str(rank),
                       "WORLD_SIZE": str(world), "LOCAL_RANK": str(rank), "MIXFP4_BENCH_BACKEND": "gloo"})
    sys.path.insert(0, ROOT)
    try:
        import torch.distributed as dist
        import bench
        r, w, local = bench.dist_setup(world)
        bench.barrier()
        step_ms = 10.0 + 5.0 * r                       # rank 1 is the slower one
        mx = bench.reduce_max(step_ms, "cpu")
        rate = bench.job_rate(100.0, w, mx)            # 100 units of work per rank
        out = io.StringIO()
        with redirect_stdout(out):                     # reference arm: only rank 0 works and prints
            if r != 0:
                bench.main(["--impl", "reference", "--steps", "3", "--warmup", "3"])
        bench.barrier()
        dist.destroy_process_group()
        q.put((r, w, local, mx, rate, out.getvalue()))
    except Exception as e:  # reported to the parent
        q.put((rank, "error", repr(e)))


def test_two_gloo_ranks_replica_bookkeeping():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank_main, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    res = [q.get(timeout=120) for _ in procs]
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    assert all(x[1] != "error" for x in res), res
    res.sort()
    for r, (rank, w, local, mx, rate, printed) in enumerate(res):
        assert (rank, w, local) == (r, 2, r)
        assert mx == 15.0                               # the slowest rank's time on every rank
        assert rate == pytest.approx(2 * 100.0 / 15e-3)  # all ranks' work over that time
    assert res[1][5] == ""                              # rank 1 of the reference arm printed nothing


def test_single_process_is_identity():
    sys.path.insert(0, ROOT)
    import bench
    assert bench.reduce_max(3.5, "cpu") == 3.5
    assert bench.job_rate(10.0, 1, 1000.0) == pytest.approx(10.0)
