"""The sharded (ZeRO-3 style) design of the path on one GPU: P emulated
ranks, each with its own context over a contiguous shard of every tensor of
the Llama-3.2-1B layout, against one unsharded context over the whole
tensors.

Each rank measures its shard (Eq. 1).  The host then adds the ranks' 3N
sums in rank order, which is what the all-reduce of the multi-rank path does,
and every rank selects (Eq. 2-4, §3.3) on the global sums.  The weights sit on
a 2^-10 grid of small integers, so every partial sum is exact in fp32 and in
fp64: the combined sums must equal the unsharded context's bit for bit, and
so must u and the masks.  The oracle's sums of sampled layers must equal them
as well, and each rank's packed block of a persisted layer (§3.1) must equal
the oracle's block of that rank's shards.
"""
import numpy as np
import pytest

from lc_workloads import gen
from lc_workloads.configs import WORKLOADS
from oracle import oracle as O
from tests.lc_harness import require_gpu

pytestmark = [pytest.mark.gpu, pytest.mark.slow]

UNIT = 2.0 ** -10


def _grid_step(torch, st, probs, seed, t):
    """W += (changed ? +-1 or +-2 : 0) units, each element changed with its
    layer's probability; R = W in units of 2^-10 at t = 0."""
    g = torch.Generator(device="cuda").manual_seed(seed * 1000 + t)
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


@pytest.mark.parametrize("ranks", [2, 3, 8])
def test_sharded_ranks_decide_like_unsharded(ranks):
    torch = require_gpu()
    import paper_2609_27193_gb300 as P
    wl = WORKLOADS["1b"]
    spec = wl.shape()
    st = gen.SyntheticState(spec, device="cuda", seed=3, master=False)
    nl = spec.nlayers
    rng = np.random.default_rng(ranks)
    probs = rng.permutation(np.geomspace(1e-4, 3e-2, nl))
    _grid_step(torch, st, probs, ranks, 0)

    def shard(k, r):
        n = st.specs[k].numel
        return n * r // ranks, n * (r + 1) // ranks

    full = P.LayerCheck()
    full.register_layout([P.segment(s.layer, st.W[k], st.R[k], st.m[k], st.v[k])
                          for k, s in enumerate(st.specs)], nl)
    full_sums = torch.zeros(3 * nl, dtype=torch.float64, device="cuda")
    full.set_layer_sums_buffer(full_sums)
    lcs, sums = [], []
    for r in range(ranks):
        segs = []
        for k, s in enumerate(st.specs):
            lo, hi = shard(k, r)
            segs.append(P.segment(s.layer, st.W[k][lo:hi], st.R[k][lo:hi], st.m[k][lo:hi],
                                  st.v[k][lo:hi]))
        lc = P.LayerCheck()
        lc.register_layout(segs, nl)
        buf = torch.zeros(3 * nl, dtype=torch.float64, device="cuda")
        lc.set_layer_sums_buffer(buf)
        lcs.append(lc)
        sums.append(buf)

    tau, K = wl.tau, wl.max_staleness
    persisted = 0
    for t in range(1, 4):
        _grid_step(torch, st, probs, ranks, t)
        full.measure(t)
        for lc in lcs:
            lc.measure(t)
        torch.cuda.synchronize()
        tot = np.zeros(3 * nl)
        for buf in sums:               # the all-reduce, in rank order
            tot += buf.cpu().numpy()
        ref = full_sums.cpu().numpy()
        assert np.array_equal(tot, ref), "combined shard sums differ from the unsharded sums"
        for buf in sums:
            buf.copy_(torch.from_numpy(tot))
        mask, u, nbytes = full.select(tau, K)
        # the oracle on the whole tensors of three layers
        for l in (0, int(np.argmax(probs)), nl - 1):
            ts = [O.Tensor(st.host("W", k), st.host("R", k))
                  for k, s in enumerate(st.specs) if s.layer == l]
            assert list(O.layer_sums(ts)) == ref[3 * l:3 * l + 3].tolist(), (t, l)
            assert u[l] == O.update_measure(*ref[3 * l:3 * l + 3], 1e-8)
        decisions = [lc.select(tau, K) for lc in lcs]
        for r, (m_r, u_r, _) in enumerate(decisions):
            assert np.array_equal(m_r, mask), "rank %d mask at step %d" % (r, t)
            assert np.array_equal(u_r, u), "rank %d u at step %d" % (r, t)
            assert lcs[r].info()["max_staleness"] == full.info()["max_staleness"]
        assert 0 < mask.sum() < nl, mask
        persisted += int(mask.sum())
        # every rank packs its shards; check the smallest persisted layer of
        # the first and the last rank against the oracle's block
        sel = np.flatnonzero(mask)
        sizes = [sum(s.numel for s in st.specs if s.layer == l) for l in sel]
        l_chk = int(sel[int(np.argmin(sizes))])
        for r, lc in enumerate(lcs):
            dst = torch.empty(max(16, lc.info()["bytes"]), dtype=torch.uint8, device="cuda")
            lc.pack_device(dst)
            lc.commit_snapshot()
            if r in (0, ranks - 1):
                torch.cuda.synchronize()
                ts = []
                for k, s in enumerate(st.specs):
                    if s.layer == l_chk:
                        lo, hi = shard(k, r)
                        ts.append(O.Tensor(st.host("W", k)[lo:hi], None, st.host("m", k)[lo:hi],
                                           st.host("v", k)[lo:hi]))
                block = O.pack_layer(ts, 256)
                off = int(lc.offsets()[l_chk])
                assert np.array_equal(dst[off:off + block.size].cpu().numpy(), block), (t, r, l_chk)
            del dst
        full.pack_device(torch.empty(max(16, nbytes), dtype=torch.uint8, device="cuda"))
        full.commit_snapshot()
        torch.cuda.synchronize()
    assert persisted > 0
    for lc in lcs:
        lc.close()
    full.close()
    del st
    torch.cuda.empty_cache()
