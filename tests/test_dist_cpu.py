"""The benchmark's multi-process path on the host (world size 2, gloo): the
barrier, the maximum over ranks of the timed region, the whole-job rate
(replicas: every rank's units over the slowest rank's time), and the
reference arm running on rank 0 only."""
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


def _rank_main(rank: int, world: int, port: int, out):
    try:
        os.environ.update({"MASTER_ADDR": "127.0.0.1", "MASTER_PORT": str(port),
                           "RANK": str(rank), "WORLD_SIZE": str(world), "LOCAL_RANK": str(rank)})
        sys.path.insert(0, ROOT)
        import bench
        w, r, local = bench.dist_env()
        d = bench.Dist(w, r, local, backend="gloo")
        d.barrier()
        # rank 1 is the slower replica: both ranks see its time
        slowest = d.max(10.0 * (rank + 1))
        rate = bench.whole_job_rate(100.0, world, slowest)
        printed = ""
        if rank == 1:  # the reference arm does nothing (and prints nothing) off rank 0
            buf = io.StringIO()
            with redirect_stdout(buf):
                ret = bench.run_reference(None, d)
            printed = buf.getvalue()
            assert ret is None
        d.barrier()
        d.close()
        out.put((rank, (w, r, local), slowest, rate, printed))
    except Exception as e:  # reported to the parent
        out.put((rank, "error", repr(e), None, None))


def test_replicas_world_size_2_gloo():
    ctx = mp.get_context("spawn")
    out = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank_main, args=(r, 2, port, out)) for r in range(2)]
    for p in procs:
        p.start()
    results = {}
    try:
        for _ in procs:
            rank, *rest = out.get(timeout=120)
            results[rank] = rest
    finally:
        for p in procs:
            p.join(timeout=30)
            if p.is_alive():
                p.kill()
    assert set(results) == {0, 1}
    for rank, (env, slowest, rate, printed) in results.items():
        assert env != "error", f"rank {rank}: {slowest}"
        assert env == (2, rank, rank)
        assert slowest == 20.0
        assert rate == pytest.approx(100.0 * 2 / 20e-3)
    assert results[1][3] == ""


def test_whole_job_rate_single_process():
    sys.path.insert(0, ROOT)
    import bench
    d = bench.Dist(1, 0, 0)
    d.barrier()
    assert d.max(3.5) == 3.5
    assert bench.whole_job_rate(90.0, 1, 1000.0) == pytest.approx(90.0)
