"""GPU parity of the pack (§3.1 full layer state), the snapshot commit, the
pinned-host store and the composite restore (§3.5, Eq. 8) against the
oracle, through the C ABI.  Packed bytes and restored state are compared
bit for bit."""
import numpy as np
import pytest

from lc_workloads import gen, shapes
from oracle.sim import digest
from tests.lc_harness import compare_decision, make_lc, make_oracle, require_gpu
from tests.test_gpu_measure_select import custom_shape

pytestmark = pytest.mark.gpu


def _host(st):
    return st.host_all("W"), st.host_all("m"), st.host_all("v")


def _assert_device_equals(st, comp, what="composite"):
    for k in range(len(st.specs)):
        w, m, v = comp[k]
        assert np.array_equal(st.host("W", k), w), "%s W of tensor %d" % (what, k)
        assert np.array_equal(st.host("R", k), w), "%s R of tensor %d" % (what, k)
        if st.has_moments[k]:
            assert np.array_equal(st.host("m", k), m), "%s m of tensor %d" % (what, k)
            assert np.array_equal(st.host("v", k), v), "%s v of tensor %d" % (what, k)


@pytest.mark.parametrize("engine", ["threads", "bulk"])
@pytest.mark.parametrize("align", [16, 256, 4096])
@pytest.mark.parametrize("alloc", ["separate", "flat", "skew"])
def test_pack_device_bytes_and_fused_commit(align, alloc, engine):
    torch = require_gpu()
    sizes = [(n, i % 3) for i, n in enumerate([1, 7, 4096, 9, 100003, 33, 2, 65536, 5])]
    spec = custom_shape(sizes)
    dts = ["bf16" if i % 4 else "f32" for i in range(len(sizes))]
    moments = [i != 5 for i in range(len(sizes))]
    st = gen.SyntheticState(spec, device="cuda", seed=4, alloc=alloc, dtypes=dts,
                            moments_mask=moments)
    st.drift(1, np.array([1e-2, 1e-5, 1e-2]))
    lc = make_lc(st, pack_align=align, copy_engine=engine)
    run = make_oracle(st, align=align)
    lc.measure(1)
    mask, u, nbytes = lc.select(1e-3, 100)
    ou, _ = run.measure(st.host_all("W"))
    run.select(ou, 1e-3, 100, 1)
    compare_decision(mask, u, run, ou, 1e-3)
    assert mask.tolist() == [1, 0, 1]
    W, M, V = _host(st)
    stream, offs = run.pack(run.last_mask, W, M, V, 1)
    assert nbytes == stream.size
    assert np.array_equal(lc.offsets()[mask == 1], offs[mask == 1])
    dst = torch.full((nbytes + 4096,), 0xAB, dtype=torch.uint8, device="cuda")
    lc.pack_device(dst)
    lc.commit_snapshot()
    torch.cuda.synchronize()
    got = dst.cpu().numpy()
    assert np.array_equal(got[:nbytes], stream), "packed stream differs from the oracle"
    assert np.all(got[nbytes:] == 0xAB), "pack wrote past its stream"
    # fused commit: R <- W for the persisted layers only
    run.commit(run.last_mask, W)
    for k in range(len(sizes)):
        assert np.array_equal(st.host("R", k), run.R[k]), "snapshot of tensor %d" % k
    c = lc.counters()
    assert c["copy_launches"] == 1
    assert c["bulk_copy_launches"] == (1 if engine == "bulk" else 0)
    lc.close()


@pytest.mark.parametrize("alloc", ["flat", "separate"])
@pytest.mark.parametrize("engine", ["bulk", "threads"])
def test_commit_unfused_and_accumulate_mode(engine, alloc):
    """The unfused commit, and accumulate mode (the measure also writes
    R <- W, Eq. 1 against W(t-1)) on both engines: flat buffers put every
    tensor on an odd 16-byte offset, so partial edge vectors are written
    element by element next to the bulk-stored interior."""
    torch = require_gpu()
    import paper_2609_27193_gb300 as P
    spec = shapes.tiny()
    for mode, fuse in ((P.LC_DRIFT_SNAPSHOT, False), (P.LC_DRIFT_ACCUMULATE, True)):
        st = gen.SyntheticState(spec, device="cuda", seed=6, alloc=alloc)
        lc = make_lc(st, fuse_commit=fuse, mode=mode, copy_engine=engine)
        run = make_oracle(st, mode=mode)
        scales = gen.loguniform(spec.nlayers, 1e-4, 1e-2, np.random.default_rng(1))
        for t in range(1, 7):
            st.drift(t, scales)
            lc.measure(t)
            mask, u, nbytes = lc.select(1e-3, 3)
            W = st.host_all("W")
            ou, _ = run.measure(W)
            run.select(ou, 1e-3, 3, t)
            compare_decision(mask, u, run, ou, 1e-3)
            dst = torch.empty(max(nbytes, 16), dtype=torch.uint8, device="cuda")
            lc.pack_device(dst)
            lc.commit_snapshot()
            run.commit(run.last_mask, W)
            for k in range(len(spec.tensors)):
                assert np.array_equal(st.host("R", k), run.R[k]), (mode, t, k)
        assert lc.counters()["bulk_measure_launches"] == (6 if engine == "bulk" else 0)
        lc.close()


@pytest.mark.parametrize("engine", ["threads", "bulk"])
@pytest.mark.parametrize("per_layer", [0, 1, 2])
def test_pack_async_store_and_restore_tiny(per_layer, engine):
    """The tiny workload for 20 steps (tau 1e-3, S_max 4), every step through
    the pinned store with a small staging ring (many chunks); masks, u and
    every persisted block against the oracle; then restores at several
    failure steps and compares the device state bit for bit.  Stores: a log
    (every version), newest-only (one version per layer), a ring of two."""
    torch = require_gpu()
    import paper_2609_27193_gb300 as P
    from lc_workloads.configs import WORKLOADS
    wl = WORKLOADS["tiny"]
    spec = wl.shape()
    st = gen.SyntheticState(spec, device="cuda", seed=wl.seed)
    scales = wl.layer_scales(spec)
    lc = make_lc(st, staging_bytes=2 << 20, copy_engine=engine)
    run = make_oracle(st)
    full = sum(lc.layer_block_bytes(l) for l in range(spec.nlayers))
    store = P.Store(lc, capacity_bytes=(wl.steps + 2) * full, versions_per_layer=per_layer)
    hole = None
    if per_layer in (0, 1):
        # a range of the arena kept out of use, inside the base step's stream
        hole = (full // 2 // 4096 * 4096, 1 << 20)
        store.exclude(*hole)
    # step 0: the base checkpoint, every layer (S_max = 0)
    lc.measure(0)
    mask, u, nbytes = lc.select(wl.tau, 0)
    assert mask.all() and nbytes == full
    W, M, V = _host(st)
    ou, _ = run.measure(W)
    run.select(ou, wl.tau, 0, 0)
    run.pack(mask, W, M, V, 0)
    lc.pack_async(store)
    lc.commit_snapshot()
    lc.wait_durable(0)
    run.mark_durable(0)
    arena = store.info()["arena"]
    history = {}
    for t in range(1, wl.steps + 1):
        st.drift(t, scales)
        W, M, V = _host(st)
        lc.measure(t)
        mask, u, nbytes = lc.select(wl.tau, wl.max_staleness)
        ou, _ = run.measure(W)
        run.select(ou, wl.tau, wl.max_staleness, t)
        compare_decision(mask, u, run, ou, wl.tau)
        stream, _ = run.pack(run.last_mask, W, M, V, t)
        assert nbytes == stream.size
        lc.pack_async(store)
        lc.commit_snapshot()
        run.commit(run.last_mask, W)
        lc.wait_durable(t)
        run.mark_durable(t)
        info = lc.info()
        mx, wt = run.staleness(t)
        assert info["max_staleness"] == mx <= wl.max_staleness - 1
        assert info["weighted_staleness"] == wt
        history[t] = int(mask.sum())
    # every block in the store equals the oracle's version of that (layer, step)
    odig = {(v["layer"], v["step"]): v["digest"] for v in run.versions}
    vers = store.versions()
    assert all(v["durable"] for v in vers)
    for i, v in enumerate(vers):
        assert digest(store.block(i)) == odig[(v["layer"], v["step"])], v
    if hole is not None:
        # no block overlaps the excluded range
        for v in vers:
            off = v["host_ptr"] - arena
            assert off + v["bytes"] <= hole[0] or off >= hole[0] + hole[1], (v, off, hole)
    if per_layer == 0:
        assert len(vers) == len(run.versions)
    if per_layer == 1:
        # newest-only: exactly the newest durable version of every layer
        assert sorted(v["layer"] for v in vers) == list(range(spec.nlayers))
        for l in range(spec.nlayers):
            newest = max(v["step"] for v in run.versions if v["layer"] == l)
            assert [v["step"] for v in vers if v["layer"] == l] == [newest]
    # restores
    # a ring store keeps the 2 newest versions per layer; with S_max = 4 the
    # last two steps are always covered by them
    points = ([wl.steps, wl.steps - 1] if per_layer == 2 else [wl.steps] if per_layer == 1
              else [wl.steps, 13, 7, 1, 0])
    for t_fail in points:
        steps = lc.restore(store, t_fail)
        comp, pick = run.composite(t_fail)
        assert steps.tolist() == [run.versions[p]["step"] for p in pick]
        torch.cuda.synchronize()
        _assert_device_equals(st, comp, "restore@%d" % t_fail)
    c = lc.counters()
    assert c["bulk_copy_launches"] == (c["copy_launches"] if engine == "bulk" else 0)
    store.close()
    lc.close()


def test_newest_only_store_capacity_and_crash():
    """A newest-only store (versions_per_layer = 1) refuses a capacity below
    every layer's block plus one block of each distinct size.  At that
    minimum a step that persists every layer still fits: the pack waits for
    the copy of the step's earlier layer of the same size, counts that
    version durable and reuses its predecessor's slot.  A block with no free
    slot and no earlier copy of its size in its step to wait for fails with
    LC_ERR_CAPACITY and leaves the store as it was.  While a new version is
    pending its predecessor stays in the plan (a crash then restores that
    one)."""
    torch = require_gpu()
    import paper_2609_27193_gb300 as P
    # layers 0 and 1 share a size class, layer 2 is the largest
    spec = custom_shape([(5000, 0), (5000, 1), (65536, 2)])
    st = gen.SyntheticState(spec, device="cuda", seed=9)
    lc = make_lc(st, staging_bytes=2 << 20)
    rb = [-(-lc.layer_block_bytes(l) // 4096) * 4096 for l in range(3)]
    assert rb[0] == rb[1] != rb[2]
    need = sum(rb) + rb[0] + rb[2]
    with pytest.raises(P.LCError) as e:
        P.Store(lc, capacity_bytes=need - 4096, versions_per_layer=1)
    assert e.value.status == 1
    store = P.Store(lc, capacity_bytes=need, versions_per_layer=1)
    lc.measure(0)
    lc.select(1e-3, 0)
    lc.pack_async(store)
    lc.commit_snapshot()
    lc.wait_durable(0)
    assert len(store) == 3 and store.info()["used_bytes"] == sum(lc.layer_block_bytes(l) for l in range(3))
    # every layer again, at the minimum capacity
    st.drift(1, np.full(3, 1e-2))
    lc.measure(1)
    mask, _, nbytes = lc.select(1e-3, 0)
    assert mask.all()
    step1 = [(st.host("W", k), st.host("m", k), st.host("v", k)) for k in range(3)]
    lc.pack_async(store)
    lc.commit_snapshot()
    lc.wait_durable(1)
    vers = store.versions()
    assert sorted((v["layer"], v["step"]) for v in vers) == [(0, 1), (1, 1), (2, 1)]
    assert all(v["durable"] for v in vers)
    # no slot for the largest layer's next block, and nothing of its step to wait for
    info = store.info()
    used = sorted((v["host_ptr"] - info["arena"], v["bytes"]) for v in vers)
    at = 0
    for off, nb in used:          # exclude every free slot
        if off > at:
            store.exclude(at, off - at)
        at = off + -(-nb // 4096) * 4096
    if at < info["capacity"]:
        store.exclude(at, info["capacity"] - at)
    st.drift(2, np.array([0.0, 0.0, 1e-2]))
    lc.measure(2)
    mask, _, nbytes = lc.select(1e-3, 100)
    assert mask.tolist() == [0, 0, 1]
    with pytest.raises(P.LCError) as e:
        lc.pack_async(store)
    assert e.value.status == 5
    assert sorted((v["layer"], v["step"]) for v in store.versions()) == [(0, 1), (1, 1), (2, 1)]
    lc.pack_device(torch.empty(nbytes, dtype=torch.uint8, device="cuda"))
    lc.commit_snapshot()
    # a pending version does not enter the plan before it is durable
    roomy = P.Store(lc, capacity_bytes=4 * need, versions_per_layer=1)
    lc.restore(store, 1)             # back to step 1's state everywhere
    torch.cuda.synchronize()
    for k in range(3):
        assert np.array_equal(st.host("W", k), step1[k][0]) and np.array_equal(st.host("v", k), step1[k][2])
    lc.measure(3)
    lc.select(1e-3, 0)
    lc.pack_async(roomy)
    lc.commit_snapshot()
    lc.wait_durable(3)
    st.drift(4, np.array([0.0, 0.0, 1e-2]))
    lc.measure(4)
    mask, _, _ = lc.select(1e-3, 100)
    assert mask.tolist() == [0, 0, 1]
    new_w = st.host("W", 2)
    lc.pack_async(roomy)
    lc.commit_snapshot()
    pick = roomy.plan(4)
    assert [roomy.version(int(p))["step"] for p in pick] == [3, 3, 3]
    lc.wait_durable(4)
    assert sorted((v["layer"], v["step"]) for v in roomy.versions()) == [(0, 3), (1, 3), (2, 4)]
    steps = lc.restore(roomy, 4)
    assert steps.tolist() == [3, 3, 4]
    torch.cuda.synchronize()
    assert np.array_equal(st.host("W", 2), new_w) and np.array_equal(st.host("R", 2), new_w)
    roomy.close()
    store.close()
    lc.close()


def _store_step_sizes(lc, nlayers, per_layer):
    """Block sizes of a step that persists every layer, in the order an
    empty store places them: layer order (log store), or each size class,
    largest first, with one slot per layer of the class plus a spare
    (newest-only store)."""
    blocks = [lc.layer_block_bytes(l) for l in range(nlayers)]
    if per_layer == 0:
        return blocks
    rounded = [-(-b // 4096) * 4096 for b in blocks]
    return [z for z in sorted(set(rounded), reverse=True) for _ in range(rounded.count(z) + 1)]


def _fits(sizes, ranges, cap):
    """Whether blocks of `sizes`, each at the first offset after the previous
    one that touches none of `ranges`, end within `cap`."""
    top = 0
    ranges = sorted(ranges)
    for z in sizes:
        at = top
        for a, n in ranges:
            if a + n <= at:
                continue
            if at + z <= a:
                break
            at = a + n
        if at + z > cap:
            return False
        top = at + z
    return True


def _expected_exclusions(rates, fraction, region, cap, sizes):
    """The regions lc_store_check_dma keeps out of use after one pass (its
    fastest and slowest pass then coincide): those below fraction x the
    median rate, slowest first, each unless a full step would then no
    longer fit (no guard when it did not fit before).  Returns those and the
    slow regions left in use (to be avoided)."""
    med = np.sort(rates)[rates.size // 2]
    slow = sorted((i for i in range(rates.size) if rates[i] < fraction * med), key=lambda i: (rates[i], i))
    guard = _fits(sizes, [], cap)
    taken, kept = [], []
    for i in slow:
        r = (i * region, min(region, cap - i * region))
        if guard and not _fits(sizes, taken + [r], cap):
            kept.append(r)
            continue
        taken.append(r)
    return taken, kept


def _full_step(lc, store, t):
    lc.measure(t)
    mask, _, _ = lc.select(1e-3, 0)          # staleness bound 0: every layer
    assert mask.all()
    lc.pack_async(store)
    lc.commit_snapshot()
    lc.wait_durable(t)


def _assert_outside(store, ranges):
    arena = store.info()["arena"]
    for v in store.versions():
        off = v["host_ptr"] - arena
        for h0, hn in ranges:
            assert off + v["bytes"] <= h0 or off >= h0 + hn, (v, off, h0, hn)


def test_store_check_dma_and_exclusions():
    """lc_store_check_dma times device->host copies into every region of an
    empty store's arena and excludes the slow ones (below a fraction of the
    median rate), slowest first, while a step that persists every layer
    still fits; the slow regions left in use are avoided by every placement
    that fits without them.  With fraction 0 nothing goes.  With one pass
    the excluded and avoided regions equal a host-side restatement of that
    rule over the rates it reports, a full step then packs around the
    excluded ones (and the avoided ones if it fits so), and a one-layer
    step of the log store keeps off both; with a huge fraction as many
    regions go as leave room for that step.  A log store too small
    for a full step loses every region and a pack finds no room.  Blocks
    are placed around ranges excluded by lc_store_exclude.  A store holding
    versions, and a ring store, are refused."""
    torch = require_gpu()
    import paper_2609_27193_gb300 as P
    spec = shapes.tiny()
    N = spec.nlayers
    st = gen.SyntheticState(spec, device="cuda", seed=12)
    lc = make_lc(st, staging_bytes=2 << 20)
    full = sum(lc.layer_block_bytes(l) for l in range(N))
    region = 1 << 20
    t = 0
    for per_layer in (0, 1):
        sizes = _store_step_sizes(lc, N, per_layer)
        store = P.Store(lc, capacity_bytes=4 * full, versions_per_layer=per_layer)
        cap = store.capacity
        rates, ex = store.check_dma(lc, region_bytes=region, min_fraction=0.0)
        assert ex == 0 and rates.size == -(-cap // region)
        assert np.all(np.isfinite(rates)) and np.all(rates > 0)
        store.close()
        for fraction in (1.0001, 1e9):
            store = P.Store(lc, capacity_bytes=4 * full, versions_per_layer=per_layer)
            rates, ex = store.check_dma(lc, region_bytes=region, min_fraction=fraction, passes=1)
            want, kept = _expected_exclusions(rates, fraction, region, cap, sizes)
            assert ex == sum(n for _, n in want) > 0, (fraction, ex)
            assert store.info()["excluded_bytes"] == ex
            assert store.info()["avoided_bytes"] == sum(n for _, n in kept)
            if fraction > 1e6:
                # every region was slow: no further region could go
                rest = [(i * region, min(region, cap - i * region)) for i in range(rates.size)]
                rest = [r for r in rest if r not in want]
                assert rest and not any(_fits(sizes, want + [r], cap) for r in rest)
            _full_step(lc, store, t)
            t += 1
            assert len(store) == N
            _assert_outside(store, want)
            if _fits(sizes, want + kept, cap):
                _assert_outside(store, kept)
            if per_layer == 0 and kept:
                # one layer's block keeps off the slow regions left in use
                store.clear()
                scales = np.zeros(N)
                scales[1] = 1e-2
                st.drift(1000 + t, scales)
                lc.measure(t)
                mask, _, _ = lc.select(1e-12, 1 << 20)
                assert mask.tolist() == [int(l == 1) for l in range(N)]
                lc.pack_async(store)
                lc.commit_snapshot()
                lc.wait_durable(t)
                t += 1
                assert len(store) == 1
                if _fits([lc.layer_block_bytes(1)], want + kept, cap):
                    _assert_outside(store, want + kept)
            store.close()
        # known holes: one inside the base step's stream, one past it
        store = P.Store(lc, capacity_bytes=4 * full, versions_per_layer=per_layer)
        holes = [(full // 2 // 4096 * 4096, 1 << 20), (2 * full // 4096 * 4096, 3 << 20)]
        for h in holes:
            store.exclude(*h)
        info = store.info()
        assert info["excluded_bytes"] == sum(h[1] for h in holes)
        _full_step(lc, store, t)
        t += 1
        vers = store.versions()
        assert len(vers) == N and store.info()["used_bytes"] == full
        _assert_outside(store, holes)
        with pytest.raises(P.LCError) as e:
            store.check_dma(lc, region_bytes=region)
        assert e.value.status == 2
        with pytest.raises(P.LCError) as e:
            store.exclude(vers[0]["host_ptr"] - info["arena"], 4096)     # a block lies there
        assert e.value.status == 2
        store.close()
    # a log store that cannot take a full step: no guard, every region goes
    small = P.Store(lc, capacity_bytes=full // 2)
    small.check_dma(lc, region_bytes=region, min_fraction=1e9)
    assert small.info()["excluded_bytes"] == small.capacity
    lc.measure(t)
    lc.select(1e-3, 0)
    t += 1
    with pytest.raises(P.LCError) as e:
        lc.pack_async(small)
    assert e.value.status == 5
    lc.pack_device(torch.empty(full, dtype=torch.uint8, device="cuda"))
    lc.commit_snapshot()
    small.close()
    ring = P.Store(lc, versions_per_layer=2)
    with pytest.raises(P.LCError) as e:
        ring.exclude(0, 4096)
    assert e.value.status == 1
    ring.close()
    lc.close()


def test_copy_trace_spans():
    """The copy trace of a staged pack and a restore: one gather span and
    one D2H span per staging chunk (one H2D and one scatter per chunk on
    the way back), covering the stream's bytes, each D2H starting after its
    chunk's gather ended (each scatter after its H2D)."""
    torch = require_gpu()
    import paper_2609_27193_gb300 as P
    spec = shapes.tiny()
    st = gen.SyntheticState(spec, device="cuda", seed=3)
    lc = make_lc(st, staging_bytes=2 << 20)
    slot = ((2 << 20) // 2) & ~4095
    full = sum(lc.layer_block_bytes(l) for l in range(spec.nlayers))
    store = P.Store(lc, capacity_bytes=2 * full)
    lc.trace_copies(True)
    lc.measure(0)
    _, _, nbytes = lc.select(1e-3, 0)
    lc.pack_async(store)
    lc.commit_snapshot()
    lc.wait_durable(0)
    spans, dropped = lc.copy_trace()
    assert dropped == 0
    nchunks = -(-nbytes // slot)
    for first, second in (("gather", "d2h"),):
        a = [x for x in spans if x["kind"] == first]
        b = [x for x in spans if x["kind"] == second]
        assert len(a) == len(b) == nchunks
        assert [x["chunk"] for x in a] == list(range(nchunks)) == [x["chunk"] for x in b]
        assert sum(x["bytes"] for x in a) == nbytes == sum(x["bytes"] for x in b)
        for x, y in zip(a, b):
            assert x["end_ms"] >= x["start_ms"] and y["end_ms"] >= y["start_ms"]
            assert y["start_ms"] >= x["end_ms"] - 0.01, (x, y)
    lc.trace_copies(True)       # clears the record
    lc.restore(store, 0)
    spans, _ = lc.copy_trace()
    h = [x for x in spans if x["kind"] == "h2d"]
    sc = [x for x in spans if x["kind"] == "scatter"]
    assert len(h) == len(sc) == -(-full // slot) and all(x["step"] == 0 for x in h)
    for x, y in zip(h, sc):
        assert y["start_ms"] >= x["end_ms"] - 0.01, (x, y)
    lc.trace_copies(False)
    assert lc.copy_trace() == ([], 0)
    store.close()
    lc.close()


def test_crash_before_durable_and_plan():
    torch = require_gpu()
    import paper_2609_27193_gb300 as P
    spec = custom_shape([(5000, 0), (777, 1), (65536, 2)])
    st = gen.SyntheticState(spec, device="cuda", seed=9)
    lc = make_lc(st, staging_bytes=2 << 20)
    store = P.Store(lc, capacity_bytes=64 << 20)
    base = [(st.host("W", k), st.host("m", k), st.host("v", k)) for k in range(3)]
    lc.measure(0)
    lc.select(1e-3, 0)
    lc.pack_async(store)
    lc.commit_snapshot()
    lc.wait_durable(0)
    st.drift(1, np.full(3, 1e-2))
    lc.measure(1)
    mask, _, _ = lc.select(1e-3, 100)
    assert mask.all()
    lc.pack_async(store)
    lc.commit_snapshot()
    # "crash": step 1 never confirmed durable -> the plan ignores it
    pick = store.plan(1)
    assert [store.version(int(p))["step"] for p in pick] == [0, 0, 0]
    torch.cuda.synchronize()
    with pytest.raises(P.LCError) as e:
        store.plan(-1)
    assert e.value.status == 7
    with pytest.raises(P.LCError) as e:
        store.clear()                  # a version is still pending
    assert e.value.status == 2
    lc.wait_durable(1)
    with pytest.raises(P.LCError) as e:
        lc.wait_durable(1)             # nothing pending any more
    assert e.value.status == 7
    lc.restore(store, 0)
    torch.cuda.synchronize()
    for k in range(3):
        assert np.array_equal(st.host("W", k), base[k][0])
        assert np.array_equal(st.host("R", k), base[k][0])
        assert np.array_equal(st.host("m", k), base[k][1])
        assert np.array_equal(st.host("v", k), base[k][2])
    # after the restore the next step continues from t_fail + 1
    lc.measure(1)
    mask, u, _ = lc.select(1e-3, 100)
    assert np.all(u == 0.0)
    store.close()
    lc.close()


def test_store_capacity_and_layout_checks():
    torch = require_gpu()
    import paper_2609_27193_gb300 as P
    spec = custom_shape([(4096, 0), (4096, 1)])
    st = gen.SyntheticState(spec, device="cuda", seed=1)
    lc = make_lc(st)
    store = P.Store(lc, capacity_bytes=1024)
    lc.measure(0)
    lc.select(1e-3, 0)
    with pytest.raises(P.LCError) as e:
        lc.pack_async(store)
    assert e.value.status == 5
    lc.pack_device(torch.empty(1 << 20, dtype=torch.uint8, device="cuda"))
    lc.commit_snapshot()
    st2 = gen.SyntheticState(custom_shape([(100, 0), (100, 1)]), device="cuda", seed=1)
    lc2 = make_lc(st2)
    with pytest.raises(P.LCError) as e:
        lc2.measure(0)
        lc2.select(1e-3, 0)
        lc2.pack_async(store)           # store built for another layout
    assert e.value.status == 1
    store.close()
    lc.close()
    lc2.close()


def test_pack_into_pinned_host_memory_directly():
    """lc_pack_device also accepts pinned host memory: the gather writes the
    packed stream straight into it over the host link (on the thread
    engine, even when the bulk engine is asked for)."""
    torch = require_gpu()
    spec = shapes.tiny()
    st = gen.SyntheticState(spec, device="cuda", seed=3)
    st.drift(1, np.full(spec.nlayers, 1e-2))
    lc = make_lc(st, copy_engine="bulk")
    run = make_oracle(st)
    lc.measure(1)
    mask, u, nbytes = lc.select(1e-3, 100)
    W, M, V = _host(st)
    ou, _ = run.measure(W)
    run.select(ou, 1e-3, 100, 1)
    compare_decision(mask, u, run, ou, 1e-3)
    stream, _ = run.pack(run.last_mask, W, M, V, 1)
    host = torch.empty(nbytes, dtype=torch.uint8, pin_memory=True)
    lc.pack_device(host)
    lc.commit_snapshot()
    torch.cuda.synchronize()
    assert np.array_equal(host.numpy(), stream)
    # host memory is never handed to the bulk engine
    assert lc.counters()["bulk_copy_launches"] == 0
    lc.close()


@pytest.mark.parametrize("alloc", ["separate", "skew"])
def test_bulk_engine_long_ranges(alloc):
    """The tiny workload packed whole with both engines: every CTA streams
    many 32 KB chunks through its ring and entries straddle CTA ranges;
    "skew" puts every snapshot one element off 16-byte alignment, so the W
    sections (whose fused commit writes the snapshot) take the thread path
    inside the bulk kernel while the moments take the bulk path.  Streams
    and snapshots against the oracle, and the two engines against each
    other."""
    torch = require_gpu()
    spec = shapes.tiny()
    out = {}
    for engine in ("bulk", "threads"):
        st = gen.SyntheticState(spec, device="cuda", seed=12, alloc=alloc)
        st.drift(1, np.full(spec.nlayers, 1e-2))
        lc = make_lc(st, copy_engine=engine)
        run = make_oracle(st)
        lc.measure(1)
        mask, u, nbytes = lc.select(1e-3, 100)
        W, M, V = _host(st)
        ou, _ = run.measure(W)
        run.select(ou, 1e-3, 100, 1)
        compare_decision(mask, u, run, ou, 1e-3)
        assert mask.all()
        stream, _ = run.pack(run.last_mask, W, M, V, 1)
        dst = torch.full((nbytes + 512,), 0x5A, dtype=torch.uint8, device="cuda")
        lc.pack_device(dst)
        lc.commit_snapshot()
        torch.cuda.synchronize()
        got = dst.cpu().numpy()
        assert np.array_equal(got[:nbytes], stream), engine
        assert np.all(got[nbytes:] == 0x5A), engine
        run.commit(run.last_mask, W)
        for k in range(len(spec.tensors)):
            assert np.array_equal(st.host("R", k), run.R[k]), (engine, k)
        c = lc.counters()
        assert c["bulk_copy_launches"] == (1 if engine == "bulk" else 0)
        out[engine] = got[:nbytes]
        lc.close()
    assert np.array_equal(out["bulk"], out["threads"])


def test_bulk_engine_wait_bound_reports_timeout():
    """LC_DEBUG_BULK_STALL makes each CTA of a bulk copy wait for 16 bytes
    that never arrive.  The bounded wait runs out (1 s), the launch returns
    after its first wave (the later waves see the fault word and stop), and
    the host reads the context's copy-fault word: lc_wait_durable and
    every later lc_select fail with LC_ERR_TIMEOUT.  The CUDA context stays
    usable: a fresh library context on the same state packs correctly."""
    import time
    torch = require_gpu()
    import paper_2609_27193_gb300 as P
    spec = shapes.tiny()
    st = gen.SyntheticState(spec, device="cuda", seed=2)
    st.drift(1, np.full(spec.nlayers, 1e-2))
    lc = make_lc(st, copy_engine="bulk", debug_flags=P.LC_DEBUG_BULK_STALL)
    store = P.Store(lc, versions_per_layer=2)
    lc.measure(1)
    mask, u, nbytes = lc.select(1e-3, 100)
    assert nbytes > 0
    t0 = time.perf_counter()
    lc.pack_async(store)
    lc.commit_snapshot()
    with pytest.raises(P.LCError) as e:
        lc.wait_durable(1)
    assert e.value.status == 6
    # eight waves of CTAs: the first gives up after its 1 s bound, the later
    # waves read the device copy of the fault word and end at once
    assert time.perf_counter() - t0 < 4.0
    assert lc.counters()["bulk_copy_launches"] == 1
    lc.measure(2)
    with pytest.raises(P.LCError) as e:
        lc.select(1e-3, 100)
    assert e.value.status == 6
    store.close()
    lc.close()
    x = torch.arange(1 << 20, device="cuda", dtype=torch.float64)
    assert float(x.sum()) == float((1 << 20) * ((1 << 20) - 1) // 2)
    st2 = gen.SyntheticState(spec, device="cuda", seed=2)
    st2.drift(1, np.full(spec.nlayers, 1e-2))
    lc2 = make_lc(st2, copy_engine="bulk")
    run = make_oracle(st2)
    lc2.measure(1)
    mask, u, nbytes = lc2.select(1e-3, 100)
    W, M, V = _host(st2)
    ou, _ = run.measure(W)
    run.select(ou, 1e-3, 100, 1)
    stream, _ = run.pack(run.last_mask, W, M, V, 1)
    dst = torch.empty(nbytes, dtype=torch.uint8, device="cuda")
    lc2.pack_device(dst)
    torch.cuda.synchronize()
    assert np.array_equal(dst.cpu().numpy(), stream)
    assert lc2.counters()["bulk_copy_launches"] == 1
    lc2.close()
