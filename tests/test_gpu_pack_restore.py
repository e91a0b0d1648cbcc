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
@pytest.mark.parametrize("per_layer", [0, 2])
def test_pack_async_store_and_restore_tiny(per_layer, engine):
    """The tiny workload for 20 steps (tau 1e-3, S_max 4), every step through
    the pinned store with a small staging ring (many chunks); masks, u and
    every persisted block against the oracle; then restores at several
    failure steps and compares the device state bit for bit."""
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
    if per_layer == 0:
        assert len(vers) == len(run.versions)
    # restores
    # a ring store keeps the 2 newest versions per layer; with S_max = 4 the
    # last two steps are always covered by them
    points = [wl.steps, wl.steps - 1] if per_layer else [wl.steps, 13, 7, 1, 0]
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
    that never arrive.  The bounded wait runs out (1 s), the launch returns,
    and the host reads the context's copy-fault word: lc_wait_durable and
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
    assert time.perf_counter() - t0 < 30.0
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
