"""The multi-process replica bookkeeping of bench.py, on CPU with gloo
(world size 2): barrier, max over ranks, whole-job rate."""
import os
import socket
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    p = s.getsockname()[1]
    s.close()
    return p


def _worker(rank, world, port, q):
    os.environ.update({"WORLD_SIZE": str(world), "RANK": str(rank), "LOCAL_RANK": str(rank),
                       "MASTER_ADDR": "127.0.0.1", "MASTER_PORT": str(port)})
    sys.path.insert(0, ROOT)
    from paper_2608_21607_gb300.replicas import Replicas
    rep = Replicas(backend="gloo")
    rep.barrier()
    seconds = 1.0 + rank              # rank 1 is the slowest
    rate, tmax = rep.job_rate(units_per_rank=100.0, seconds_this_rank=seconds)
    q.put((rank, rep.world, rate, tmax, rep.max(10 * rank)))
    rep.close()


def test_replicas_gloo_world2():
    import torch.multiprocessing as mp
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    out = sorted(q.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    for rank, world, rate, tmax, mx in out:
        assert world == 2
        assert tmax == pytest.approx(2.0)          # the slowest rank's time
        assert rate == pytest.approx(2 * 100.0 / 2.0)
        assert mx == pytest.approx(10.0)


def test_single_process_defaults(monkeypatch):
    monkeypatch.delenv("WORLD_SIZE", raising=False)
    sys.path.insert(0, ROOT)
    from paper_2608_21607_gb300.replicas import Replicas
    rep = Replicas()
    assert rep.world == 1 and rep.dist is None
    rate, t = rep.job_rate(50.0, 2.0)
    assert rate == 25.0 and t == 2.0
