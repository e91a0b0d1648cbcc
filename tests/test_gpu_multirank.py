"""The multi-rank path through the library in real processes (§4.1: under
ZeRO-3 each rank holds a shard of every layer and checkpoints it on its own).

Two processes share cuda:0.  Each owns a library context over its half of
every tensor of the Llama-3.2-1B layout and keeps the per-layer sums in a
tensor it owns (lc_set_layer_sums_buffer).  Between lc_measure and
lc_select it all-reduces that tensor with torch.distributed (gloo) on the
library's stream, then selects and packs its shards.  The kernels of the two
processes never wait on each other: the only exchange is the host-side
all-reduce.

The weights sit on a 2^-10 grid of small integers, so every partial sum is
exact: after the all-reduce each rank's sums, u and mask must equal those of
one unsharded context over the whole tensors bit for bit (rank 0 runs it),
the oracle's sums of sampled layers must equal them, and each rank's packed
block of a persisted layer (§3.1) must equal the oracle's block of that
rank's shards.
"""
import datetime
import os
import socket
import traceback

import numpy as np
import pytest

from tests.lc_harness import require_gpu

pytestmark = [pytest.mark.gpu, pytest.mark.slow]

WORLD = 2
STEPS = 3
UNIT = 2.0 ** -10


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _grid_step(torch, st, probs, t):
    """W += +-1 or +-2 units for each element changed (its layer's
    probability); W = R on the grid at t = 0.  Seeded, so every process
    draws the same tensors."""
    g = torch.Generator(device="cuda").manual_seed(7000 + t)
    for k, spec in enumerate(st.specs):
        n = spec.numel
        if t == 0:
            r = torch.randint(-8, 9, (n,), device="cuda", generator=g).float() * UNIT
            st.W[k].copy_(r)
            st.R[k].copy_(r)
            continue
        step = torch.randint(1, 3, (n,), device="cuda", generator=g).float()
        sign = torch.randint(0, 2, (n,), device="cuda", generator=g).float() * 2 - 1
        keep = torch.rand(n, device="cuda", generator=g) < probs[spec.layer]
        st.W[k].copy_(st.W[k].float() + step * sign * keep.float() * UNIT)
        del step, sign, keep


def _worker(rank, port, q):
    try:
        import torch
        import torch.distributed as dist
        os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
        dist.init_process_group("gloo", rank=rank, world_size=WORLD,
                                timeout=datetime.timedelta(seconds=120))
        torch.cuda.set_device(0)
        import paper_2609_27193_gb300 as P
        from lc_workloads import gen
        from lc_workloads.configs import WORKLOADS
        from oracle import oracle as O
        wl = WORKLOADS["1b"]
        spec = wl.shape()
        nl = spec.nlayers
        st = gen.SyntheticState(spec, device="cuda", seed=3, master=False)
        probs = np.random.default_rng(5).permutation(np.geomspace(1e-4, 3e-2, nl))
        _grid_step(torch, st, probs, 0)

        def shard(k):
            n = st.specs[k].numel
            return n * rank // WORLD, n * (rank + 1) // WORLD

        side = torch.cuda.Stream()
        lc = P.LayerCheck(device=0, stream=side)
        segs = []
        for k, s in enumerate(st.specs):
            lo, hi = shard(k)
            segs.append(P.segment(s.layer, st.W[k][lo:hi], st.R[k][lo:hi], st.m[k][lo:hi], st.v[k][lo:hi]))
        lc.register_layout(segs, nl)
        sums = torch.zeros(3 * nl, dtype=torch.float64, device="cuda")
        lc.set_layer_sums_buffer(sums)
        full = full_sums = None
        if rank == 0:
            full = P.LayerCheck(device=0)
            full.register_layout([P.segment(s.layer, st.W[k], st.R[k], st.m[k], st.v[k])
                                  for k, s in enumerate(st.specs)], nl)
            full_sums = torch.zeros(3 * nl, dtype=torch.float64, device="cuda")
            full.set_layer_sums_buffer(full_sums)
        torch.cuda.synchronize()
        tau, K = wl.tau, wl.max_staleness
        persisted = 0
        for t in range(1, STEPS + 1):
            _grid_step(torch, st, probs, t)
            torch.cuda.synchronize()
            lc.measure(t)
            with torch.cuda.stream(side):
                dist.all_reduce(sums)          # the library's stream: measure -> all-reduce -> select
            mask, u, nbytes = lc.select(tau, K)
            got = sums.cpu().numpy()
            # every rank's decision against rank 0's unsharded context
            dec = torch.from_numpy(np.concatenate([u, mask.astype(np.float64), got]))
            gathered = [torch.zeros_like(dec) for _ in range(WORLD)]
            dist.all_gather(gathered, dec)
            if rank == 0:
                full.measure(t)
                fmask, fu, _ = full.select(tau, K)
                ref = full_sums.cpu().numpy()
                for r, g_r in enumerate(gathered):
                    g_r = g_r.numpy()
                    assert np.array_equal(g_r[2 * nl:], ref), "rank %d sums at step %d" % (r, t)
                    assert np.array_equal(g_r[:nl], fu), "rank %d u at step %d" % (r, t)
                    assert np.array_equal(g_r[nl:2 * nl], fmask.astype(np.float64)), "rank %d mask" % r
                for l in (0, int(np.argmax(probs)), nl - 1):
                    ts = [O.Tensor(st.host("W", k), st.host("R", k))
                          for k, s in enumerate(st.specs) if s.layer == l]
                    assert list(O.layer_sums(ts)) == ref[3 * l:3 * l + 3].tolist(), (t, l)
                assert 0 < fmask.sum() < nl, fmask
            persisted += int(mask.sum())
            dst = torch.empty(max(16, nbytes), dtype=torch.uint8, device="cuda")
            lc.pack_device(dst)
            lc.commit_snapshot()
            side.synchronize()
            sel = np.flatnonzero(mask)
            sizes = [sum(s.numel for s in st.specs if s.layer == l) for l in sel]
            l_chk = int(sel[int(np.argmin(sizes))])
            ts = []
            for k, s in enumerate(st.specs):
                if s.layer == l_chk:
                    lo, hi = shard(k)
                    ts.append(O.Tensor(st.host("W", k)[lo:hi], None, st.host("m", k)[lo:hi],
                                       st.host("v", k)[lo:hi]))
            block = O.pack_layer(ts, 256)
            off = int(lc.offsets()[l_chk])
            assert np.array_equal(dst[off:off + block.size].cpu().numpy(), block), (rank, t, l_chk)
            del dst
            if rank == 0:
                fb = full.info()["bytes"]
                full.pack_device(torch.empty(max(16, fb), dtype=torch.uint8, device="cuda"))
                full.commit_snapshot()
            torch.cuda.synchronize()
            dist.barrier()
        launches = lc.counters()["kernel_launches"]
        lc.close()
        if full is not None:
            full.close()
        dist.destroy_process_group()
        q.put((rank, "ok", persisted, launches))
    except BaseException:
        q.put((rank, traceback.format_exc(), 0, 0))


def test_two_processes_all_reduce_the_sums_between_measure_and_select():
    require_gpu()
    import torch.multiprocessing as mp
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, port, q)) for r in range(WORLD)]
    for p in procs:
        p.start()
    results = []
    try:
        for _ in range(WORLD):
            results.append(q.get(timeout=600))
    finally:
        for p in procs:
            p.join(timeout=60)
            if p.is_alive():
                p.kill()
                p.join()
    errors = [r for r in results if r[1] != "ok"]
    assert not errors, "\n".join("rank %d:\n%s" % (r[0], r[1]) for r in errors)
    assert sorted(r[0] for r in results) == list(range(WORLD))
    for _, _, persisted, launches in results:
        assert persisted > 0
        # per step: one measure, one select, one pack
        assert launches == 3 * STEPS
