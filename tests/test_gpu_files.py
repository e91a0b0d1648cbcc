"""§3.5 recovery from the file tier on the GPU: the tiny workload persists
through a pinned store, every durable version is appended to a checkpoint
directory, and a fresh context recovers from the directory alone.  The
records the library wrote are read back by the independent reader
(oracle/files.py) and the blocks compared with the oracle's versions; the
device state after lc_store_load_dir + lc_restore equals the oracle's
composite bit for bit at several failure steps; a damaged newest block
makes the recovery fall back to the layer's previous version."""
import os

import numpy as np
import pytest

from lc_workloads import gen
from lc_workloads.configs import WORKLOADS
from oracle import files as F
from oracle.sim import digest
from tests.lc_harness import make_lc, make_oracle, require_gpu

pytestmark = pytest.mark.gpu


def _device_equals(st, comp, what):
    for k in range(len(st.specs)):
        w, m, v = comp[k]
        assert np.array_equal(st.host("W", k), w), "%s W of tensor %d" % (what, k)
        assert np.array_equal(st.host("R", k), w), "%s R of tensor %d" % (what, k)
        if st.has_moments[k]:
            assert np.array_equal(st.host("m", k), m), "%s m of tensor %d" % (what, k)
            assert np.array_equal(st.host("v", k), v), "%s v of tensor %d" % (what, k)


def test_persist_dir_and_metadata_driven_restore(tmp_path):
    torch = require_gpu()
    import paper_2609_27193_gb300 as P
    wl = WORKLOADS["tiny"]
    spec = wl.shape()
    st = gen.SyntheticState(spec, device="cuda", seed=wl.seed)
    scales = wl.layer_scales(spec)
    lc = make_lc(st)
    run = make_oracle(st)
    layer_bytes = [lc.layer_block_bytes(l) for l in range(spec.nlayers)]
    store = P.Store(lc, versions_per_layer=2)       # a ring: the directory keeps the history
    d = str(tmp_path / "ckpt")
    written = 0
    steps = 12
    for t in range(0, steps + 1):
        if t:
            st.drift(t, scales)
        W, M, V = st.host_all("W"), st.host_all("m"), st.host_all("v")
        lc.measure(t)
        mask, u, nbytes = lc.select(wl.tau, wl.max_staleness if t else 0)
        ou, _ = run.measure(W)
        run.select(ou, wl.tau, wl.max_staleness if t else 0, t)
        assert np.array_equal(mask, run.last_mask)
        run.pack(run.last_mask, W, M, V, t)
        lc.pack_async(store)
        lc.commit_snapshot()
        run.commit(run.last_mask, W)
        lc.wait_durable(t)
        run.mark_durable(t)
        written += store.persist_dir(d, sync=(t == steps))
    assert store.persist_dir(d) == 0                 # nothing new: idempotent
    nl, lay, recs, torn = F.read_dir(d)
    assert nl == spec.nlayers and lay == F.layout_crc(layer_bytes) and not torn
    assert [(r["layer"], r["step"]) for r in recs] == [(v["layer"], v["step"]) for v in run.versions]
    assert written == sum(r["bytes"] for r in recs)
    for r, v in zip(recs, run.versions):
        blk = F.read_block(d, r)
        assert digest(blk) == v["digest"], (r["layer"], r["step"])
        if r["bytes"] <= (64 << 10):
            assert F.crc32c(blk.tobytes()) == r["block_crc"]
    got, _, _, _ = P.manifest_read(d, verify_blocks=True)
    assert all(g["intact"] for g in got)
    store.close()
    lc.close()

    # recovery in a fresh context over different device contents
    st2 = gen.SyntheticState(spec, device="cuda", seed=wl.seed + 1)
    lc2 = make_lc(st2)
    for t_fail in (steps, 7, 3, 0):
        ld, lsteps = lc2.load_dir(d, t_fail)
        pick = F.pick(recs, layer_bytes, t_fail)
        assert lsteps.tolist() == [recs[i]["step"] for i in pick]
        assert lc2.restore(ld, t_fail).tolist() == lsteps.tolist()
        torch.cuda.synchronize()
        comp, opick = run.composite(t_fail)
        assert [run.versions[i]["step"] for i in opick] == lsteps.tolist()
        _device_equals(st2, comp, "restore@%d" % t_fail)
        ld.close()

    # a damaged newest block: that layer falls back to its previous version
    newest = max(range(len(recs)), key=lambda i: (recs[i]["step"], i))
    l = recs[newest]["layer"]
    with open(os.path.join(d, "blocks.lcb"), "r+b") as f:
        f.seek(recs[newest]["offset"] + 5)
        b = f.read(1)
        f.seek(recs[newest]["offset"] + 5)
        f.write(bytes([b[0] ^ 0x10]))
    ld, lsteps = lc2.load_dir(d, steps)
    prev = max((i for i, r in enumerate(recs) if r["layer"] == l and i != newest),
               key=lambda i: (recs[i]["step"], i))
    assert lsteps[l] == recs[prev]["step"] < recs[newest]["step"]
    lc2.restore(ld, steps)
    torch.cuda.synchronize()
    run.versions[newest]["durable"] = False          # the oracle's view: that version is gone
    comp, _ = run.composite(steps)
    _device_equals(st2, comp, "restore past a damaged block")
    ld.close()
    # a torn manifest tail is ignored by the reader and cut by the next append
    with open(os.path.join(d, "manifest.lcm"), "ab") as f:
        f.write(b"LCVR" + bytes(20))
    _, _, _, torn = P.manifest_read(d, verify_blocks=False)
    assert torn
    ld, lsteps2 = lc2.load_dir(d, steps)
    assert lsteps2.tolist() == lsteps.tolist()
    assert ld.persist_dir(d) == 0                    # every version is on file already
    got, _, _, torn = P.manifest_read(d, verify_blocks=False)
    assert not torn and len(got) == len(recs)
    ld.close()
    with pytest.raises(P.LCError) as e:
        lc2.load_dir(d, -1)
    assert e.value.status == 7
    lc2.close()
