"""The bench's whole-job figures under several ranks, on CPU with two gloo
ranks: `value` and `e2e` are every rank's bytes over the slowest rank's
time (weak scaling), so each rank must see the sum of the bytes and the
maximum of the times."""
import datetime
import os
import socket
import sys

import pytest

torch = pytest.importorskip("torch")
import torch.distributed as dist
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, q):
    try:
        os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
        dist.init_process_group("gloo", rank=rank, world_size=world,
                                timeout=datetime.timedelta(seconds=60))
        sys.path.insert(0, ROOT)
        import bench
        # rank r moved (r + 1) * 1e12 + 1 bytes in 2.5 + r seconds
        got = bench.whole_job((rank + 1) * 1e12 + 1, 2.5 + rank, world, "cpu")
        q.put((rank, got))
        dist.destroy_process_group()
    except Exception as e:  # pragma: no cover - reported to the parent
        q.put((rank, repr(e)))


def test_whole_job_sums_bytes_and_takes_the_slowest_rank():
    world = 2
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, world, port, q)) for r in range(world)]
    for p in procs:
        p.start()
    out = dict(q.get(timeout=120) for _ in range(world))
    for p in procs:
        p.join(timeout=60)
    for r in range(world):
        assert out[r] == (3e12 + 2, 3.5), out[r]


def test_whole_job_single_rank_is_the_identity():
    sys.path.insert(0, ROOT)
    import bench
    assert bench.whole_job(12345, 0.5, 1, "cpu") == (12345.0, 0.5)
