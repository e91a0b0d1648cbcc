"""64-bit indexing: a layer whose one bf16 segment holds n = 2^31 + 4099
elements (more than an int32 counts), beside a small layer, through measure
(Eq. 1), select, the device pack (§3.1), the fused commit, the pinned store
and the composite restore (§3.5, Eq. 8).

Closed form for Eq. 1: R = 1 everywhere and W = 2 on a known set P of
positions, 1 elsewhere, so D = |P| and A = n exactly (every partial sum is an
integer: below 2^24 in an fp32 partial, below 2^53 in fp64).  P sits where a
32-bit element or byte index would wrap or truncate: around 2^30, around
2^31 and in the ragged tail.  The layer's packed block is 21.5 GB and its
exp_avg_sq section starts past 2^33 bytes; every section is compared with its
source in full on the device, and the alignment padding must be zero.
"""
import numpy as np
import pytest

from oracle import oracle as O
from tests.lc_harness import require_gpu

pytestmark = [pytest.mark.gpu, pytest.mark.slow]

N_BIG = (1 << 31) + 4099
N_SMALL = 1000
CHUNK = 1 << 28


def _fill_pattern(t, salt):
    """Writes a hash of the element index into the int32 view of t."""
    import torch
    v = t.view(torch.int32)
    for c0 in range(0, v.numel(), CHUNK):
        c1 = min(v.numel(), c0 + CHUNK)
        x = torch.arange(c0, c1, device=v.device, dtype=torch.int64)
        v[c0:c1] = ((x * 2654435761 + salt) & 0x7FFFFFFF).to(torch.int32)


def _is_pattern(t, salt):
    import torch
    v = t.view(torch.int32)
    for c0 in range(0, v.numel(), CHUNK):
        c1 = min(v.numel(), c0 + CHUNK)
        x = torch.arange(c0, c1, device=v.device, dtype=torch.int64)
        if not torch.equal(v[c0:c1], ((x * 2654435761 + salt) & 0x7FFFFFFF).to(torch.int32)):
            return False
    return True


def _check_block(blk, srcs, align):
    """blk holds one layer's packed block: the W, exp_avg and exp_avg_sq
    sections of its single segment, each padded with zeros to `align`."""
    import torch
    off = 0
    for name, t in zip(("W", "exp_avg", "exp_avg_sq"), srcs):
        nb = t.numel() * t.element_size()
        assert torch.equal(blk[off:off + nb], t.view(torch.uint8)), "section %s" % name
        padded = -(-nb // align) * align
        assert not blk[off + nb:off + padded].any(), "padding after %s" % name
        off += padded
    assert off == blk.numel()


def _w_is(w, ones_except):
    """w is 1 everywhere except at the given (index, value) pairs."""
    import torch
    idx = torch.tensor([i for i, _ in ones_except], device=w.device, dtype=torch.int64)
    val = torch.tensor([v for _, v in ones_except], device=w.device, dtype=torch.float32)
    return (int((w != 1).sum()) == len(ones_except)
            and torch.equal(w[idx].float(), val))


@pytest.mark.parametrize("engine,skew", [("bulk", 0), ("bulk", 1), ("threads", 1)])
def test_segment_beyond_int32_elements(engine, skew):
    torch = require_gpu()
    import paper_2609_27193_gb300 as P
    dev = "cuda"
    # skew = 1: W and R start 2 bytes, the moments 12 bytes past a 16-byte boundary
    wbuf = torch.ones(N_BIG + 8, dtype=torch.bfloat16, device=dev)
    rbuf = torch.ones(N_BIG + 8, dtype=torch.bfloat16, device=dev)
    mbuf = torch.empty(N_BIG + 8, dtype=torch.float32, device=dev)
    vbuf = torch.empty(N_BIG + 8, dtype=torch.float32, device=dev)
    W, R = wbuf[skew:skew + N_BIG], rbuf[skew:skew + N_BIG]
    M, V = mbuf[3 * skew:3 * skew + N_BIG], vbuf[3 * skew:3 * skew + N_BIG]
    _fill_pattern(M, 11)
    _fill_pattern(V, 23)
    g = torch.Generator(device=dev).manual_seed(5)
    w1 = (torch.randn(N_SMALL, device=dev, generator=g) * 0.02).to(torch.bfloat16)
    r1 = w1.clone()
    m1 = torch.randn(N_SMALL, device=dev, generator=g)
    v1 = torch.rand(N_SMALL, device=dev, generator=g)

    two31 = 1 << 31
    pos = sorted(set([0, 1, (1 << 30) - 1, 1 << 30, two31 - 2, two31 - 1, two31, two31 + 1]
                     + list(range(two31 - 300, two31 + 300))
                     + list(range(N_BIG - 4099, N_BIG, 97)) + [N_BIG - 1]))
    W[torch.tensor(pos, device=dev)] = 2.0
    step0_w = [(i, 2.0) for i in pos]

    lc = P.LayerCheck(copy_engine=engine)
    lc.register_layout([P.segment(0, W, R, M, V), P.segment(1, w1, r1, m1, v1)], 2)
    sums = torch.zeros(6, dtype=torch.float64, device=dev)
    lc.set_layer_sums_buffer(sums)
    b0, b1 = lc.layer_block_bytes(0), lc.layer_block_bytes(1)
    align = 256
    assert b0 == sum(-(-(N_BIG * e) // align) * align for e in (2, 4, 4)) and b0 > (1 << 34)
    store = P.Store(lc, capacity_bytes=b0 + b1 + (1 << 20))

    # step 0: every layer persists (S_max = 0)
    lc.measure(0)
    mask, u, nbytes = lc.select(1e-3, 0)
    s = sums.cpu().numpy()
    assert s[0:3].tolist() == [float(len(pos)), float(N_BIG), float(N_BIG)]
    assert u[0] == O.update_measure(len(pos), N_BIG, N_BIG, 1e-8)
    assert mask.tolist() == [1, 1] and nbytes == b0 + b1
    lc.pack_async(store)
    lc.commit_snapshot()
    lc.wait_durable(0)
    torch.cuda.synchronize()
    assert torch.equal(R.view(torch.int16), W.view(torch.int16)), "fused commit of layer 0"
    assert torch.equal(r1, w1)
    vers = store.versions()
    assert [(v["layer"], v["step"], v["bytes"]) for v in vers] == [(0, 0, b0), (1, 0, b1)]
    dst = torch.empty(b0, dtype=torch.uint8, device=dev)
    dst.copy_(torch.from_numpy(store.block(0)))
    _check_block(dst, (W, M, V), align)
    saved1 = (w1.clone(), m1.clone(), v1.clone())

    # step 1: new weights at P' (disjoint from P) and new moments in both layers
    pos1 = [5, two31 + 1001, two31 + 1002, N_BIG - 2]
    W[torch.tensor(pos1, device=dev)] = 3.0
    _fill_pattern(M, 31)
    _fill_pattern(V, 37)
    w1.add_(0.25)
    m1.mul_(-1.0)
    lc.measure(1)
    mask, u, nbytes = lc.select(1e-12, 8)
    s = sums.cpu().numpy()
    assert s[0:3].tolist() == [2.0 * len(pos1), float(N_BIG + len(pos)), float(N_BIG)]
    assert mask.tolist() == [1, 1] and nbytes == b0 + b1
    dst = torch.full((b0 + b1,), 0xAB, dtype=torch.uint8, device=dev)
    lc.pack_device(dst)
    lc.commit_snapshot()
    torch.cuda.synchronize()
    off = lc.offsets()
    assert off.tolist() == [0, b0]
    _check_block(dst[:b0], (W, M, V), align)
    _check_block(dst[b0:], (w1, m1, v1), align)
    assert torch.equal(R.view(torch.int16), W.view(torch.int16)), "fused commit at step 1"
    del dst

    # restore at t_fail = 1: only step 0 is durable in the store
    steps = lc.restore(store, 1)
    torch.cuda.synchronize()
    assert steps.tolist() == [0, 0]
    assert _w_is(W, step0_w), "restored W of layer 0"
    assert torch.equal(R.view(torch.int16), W.view(torch.int16)), "restored R of layer 0"
    assert _is_pattern(M, 11) and _is_pattern(V, 23), "restored moments of layer 0"
    for got, want in zip((w1, m1, v1), saved1):
        assert torch.equal(got, want)
    assert torch.equal(r1, w1)
    # the bytes outside the segments were never written
    assert wbuf[:skew].eq(1).all() and wbuf[skew + N_BIG:].eq(1).all()
    c = lc.counters()
    if engine == "bulk":
        assert c["bulk_copy_launches"] > 0 and c["bulk_measure_launches"] == 2
    else:
        assert c["bulk_copy_launches"] == 0 and c["bulk_measure_launches"] == 0
    store.close()
    lc.close()
    del W, R, M, V, wbuf, rbuf, mbuf, vbuf
    torch.cuda.empty_cache()
