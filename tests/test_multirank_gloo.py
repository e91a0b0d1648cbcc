"""Sharded (data-parallel) design on CPU with two gloo ranks.

Under ZeRO-3 every rank holds a shard of every layer.  Each rank computes
its shard's (D, A, n) sums of Eq. 1; one all-reduce (sum) of the 3N values
makes every rank take the same decision.  Here each rank runs the oracle on
its half of every tensor, all-reduces with gloo, and selects; the result
must equal the unsharded oracle on the whole tensors (measures within
1e-12, masks exact).  A rank that never joins makes the others fail with a
timeout instead of hanging."""
import datetime
import os
import socket

import numpy as np
import pytest

torch = pytest.importorskip("torch")
import torch.distributed as dist
import torch.multiprocessing as mp


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _inputs():
    from lc_workloads import gen, shapes
    st = gen.SyntheticState(shapes.tiny(), device="cpu", seed=11)
    st.drift(1, np.geomspace(1e-4, 3e-2, 6))
    return st


def _worker(rank, world, port, q):
    try:
        os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
        dist.init_process_group("gloo", rank=rank, world_size=world,
                                timeout=datetime.timedelta(seconds=60))
        from oracle import oracle as O
        st = _inputs()
        W, R = st.host_all("W"), st.host_all("R")
        sums = np.zeros((st.nlayers, 3))
        for l in range(st.nlayers):
            ts = []
            for k, t in enumerate(st.specs):
                if t.layer != l:
                    continue
                n = t.numel
                lo, hi = n * rank // world, n * (rank + 1) // world
                if hi > lo:
                    ts.append(O.Tensor(W[k][lo:hi], R[k][lo:hi]))
            sums[l] = O.layer_sums(ts) if ts else (0.0, 0.0, 0.0)
        buf = torch.from_numpy(sums.reshape(-1).copy())
        dist.all_reduce(buf)
        g = buf.numpy().reshape(-1, 3)
        u = np.array([O.update_measure(d, a, n, 1e-8) for d, a, n in g])
        delta = np.zeros(st.nlayers)
        tl = np.zeros(st.nlayers, dtype=np.int64)
        mask, _, _ = O.select_step(u, delta, tl, 1e-3, 4, 1)
        q.put((rank, u, mask))
        dist.destroy_process_group()
    except Exception as e:  # reported to the parent
        q.put((rank, "error", repr(e)))


def test_two_rank_allreduce_matches_unsharded():
    from oracle import oracle as O
    from oracle.sim import OracleRun
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    res = [q.get(timeout=120) for _ in procs]
    for p in procs:
        p.join(timeout=60)
    for r in res:
        assert not (isinstance(r[1], str) and r[1] == "error"), r
    st = _inputs()
    run = OracleRun(st.tensor_layer, st.numels, st.nlayers)
    run.set_reference(st.host_all("R"))
    u_ref, _ = run.measure(st.host_all("W"))
    mask_ref = run.select(u_ref, 1e-3, 4, 1)
    for rank, u, mask in res:
        assert np.all(np.abs(u - u_ref) <= 1e-12 * np.abs(u_ref))
        assert np.array_equal(mask, mask_ref)
    assert 0 < mask_ref.sum() < st.nlayers


def _lonely(rank, world, port, q):
    try:
        os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
        dist.init_process_group("gloo", rank=rank, world_size=world,
                                timeout=datetime.timedelta(seconds=3))
        q.put((rank, "joined"))
    except Exception as e:
        q.put((rank, "failed: " + type(e).__name__))


def test_missing_rank_fails_with_timeout_not_hang():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    p = ctx.Process(target=_lonely, args=(0, 2, _free_port(), q))
    p.start()
    rank, status = q.get(timeout=120)
    p.join(timeout=60)
    assert status.startswith("failed"), status
