"""Steps without a host round trip (lc_step_async / lc_step_wait) and their
CUDA-graph form (lc_step_graph_create / lc_step_graph_launch), against the
oracle in lockstep: decisions, measures, packed streams (into device or
pinned host memory) and snapshots; capacity overflow persists nothing."""
import numpy as np
import pytest

from lc_workloads import gen, shapes
from lc_workloads.configs import WORKLOADS
from oracle import oracle as O
from tests.lc_harness import compare_decision, make_lc, make_oracle, require_gpu

pytestmark = pytest.mark.gpu


def _oracle_step(run, st, t, tau, K):
    W = st.host_all("W")
    ou, _ = run.measure(W)
    run.select(ou, tau, K, t)
    return W, ou


@pytest.mark.parametrize("where", ["device", "pinned"])
def test_async_steps_lockstep_tiny(where):
    torch = require_gpu()
    wl = WORKLOADS["tiny"]
    spec = wl.shape()
    st = gen.SyntheticState(spec, device="cuda", seed=3)
    scales = wl.layer_scales(spec)
    lc = make_lc(st)
    run = make_oracle(st)
    full = sum(lc.layer_block_bytes(l) for l in range(spec.nlayers))
    dst = (torch.empty(full, dtype=torch.uint8, device="cuda") if where == "device"
           else torch.empty(full, dtype=torch.uint8, pin_memory=True))
    for t in range(1, wl.steps + 1):
        st.drift(t, scales)
        lc.step_async(t, wl.tau, wl.max_staleness, dst)
        mask, u, nbytes = lc.step_wait(t)
        W, ou = _oracle_step(run, st, t, wl.tau, wl.max_staleness)
        compare_decision(mask, u, run, ou, wl.tau)
        M, V = st.host_all("m"), st.host_all("v")
        stream, _ = run.pack(run.last_mask, W, M, V, t)
        run.commit(run.last_mask, W)
        assert nbytes == stream.size
        torch.cuda.synchronize()
        got = (dst[:nbytes].cpu() if where == "device" else dst[:nbytes]).numpy()
        assert np.array_equal(got, stream), "packed stream of step %d" % t
        for k in range(len(spec.tensors)):
            assert np.array_equal(st.host("R", k), run.R[k])
        info = lc.info()
        assert info["max_staleness"] == run.staleness(t)[0]
    lc.close()


def test_four_steps_in_flight():
    torch = require_gpu()
    import paper_2609_27193_gb300 as P
    spec = shapes.tiny()
    st = gen.SyntheticState(spec, device="cuda", seed=4)
    scales = np.geomspace(1e-4, 3e-2, spec.nlayers)
    lc = make_lc(st)
    run = make_oracle(st)
    full = sum(lc.layer_block_bytes(l) for l in range(spec.nlayers))
    dsts = [torch.empty(full, dtype=torch.uint8, device="cuda") for _ in range(4)]
    saved = []
    for t in range(1, 5):                 # everything on the current stream, no host sync
        st.drift(t, scales)
        saved.append([w.clone() for w in st.W])
        lc.step_async(t, 1e-3, 3, dsts[t - 1])
    with pytest.raises(P.LCError) as e:
        lc.step_async(5, 1e-3, 3, dsts[0])
    assert e.value.status == 2            # a fifth step would exceed the slots
    for t in range(1, 5):
        mask, u, nbytes = lc.step_wait(t)
        W = [st.to_numpy(w) for w in saved[t - 1]]
        ou, _ = run.measure(W)
        run.select(ou, 1e-3, 3, t)
        compare_decision(mask, u, run, ou, 1e-3)
        run.commit(run.last_mask, W)
    with pytest.raises(P.LCError) as e:
        lc.step_wait(2)                   # already read
    assert e.value.status == 7
    lc.close()


def test_capacity_overflow_persists_nothing():
    torch = require_gpu()
    import paper_2609_27193_gb300 as P
    spec = shapes.tiny()
    st = gen.SyntheticState(spec, device="cuda", seed=5)
    scales = np.full(spec.nlayers, 2e-2)
    lc = make_lc(st)
    run = make_oracle(st)
    small = torch.empty(4096, dtype=torch.uint8, device="cuda")
    st.drift(1, scales)
    R_before = [st.host("R", k) for k in range(len(spec.tensors))]
    lc.step_async(1, 1e-3, 100, small)
    with pytest.raises(P.LCError) as e:
        lc.step_wait(1)
    assert e.value.status == 5
    # the oracle's view of a step that persisted nothing: the drift stays accumulated
    W, ou = _oracle_step(run, st, 1, 1e-3, 100)
    acc_before, tl_before, u, _ = run._undo
    run.delta[:] = ou if run.mode == O.SNAPSHOT else acc_before + ou
    run.t_last[:] = tl_before
    for k in range(len(spec.tensors)):
        assert np.array_equal(st.host("R", k), R_before[k]), "snapshot changed on overflow"
    full = sum(lc.layer_block_bytes(l) for l in range(spec.nlayers))
    dst = torch.empty(full, dtype=torch.uint8, device="cuda")
    st.drift(2, scales)
    lc.step_async(2, 1e-3, 100, dst)
    mask, u, nbytes = lc.step_wait(2)
    W, ou = _oracle_step(run, st, 2, 1e-3, 100)
    compare_decision(mask, u, run, ou, 1e-3)
    assert mask.sum() > 0
    lc.close()


@pytest.mark.parametrize("where", ["device", "pinned"])
def test_graph_steps_lockstep(where):
    torch = require_gpu()
    import paper_2609_27193_gb300 as P
    spec = shapes.tiny()
    st = gen.SyntheticState(spec, device="cuda", seed=6)
    scales = np.geomspace(1e-4, 3e-2, spec.nlayers)
    stream = torch.cuda.Stream()
    lc = make_lc(st, stream=stream)
    run = make_oracle(st)
    full = sum(lc.layer_block_bytes(l) for l in range(spec.nlayers))
    dst = (torch.empty(full, dtype=torch.uint8, device="cuda") if where == "device"
           else torch.empty(full, dtype=torch.uint8, pin_memory=True))
    lc.step_graph_create(1e-3, 3, dst)
    # a normal step first; graph steps then continue the numbering on the device
    st.drift(1, scales)
    torch.cuda.synchronize()
    lc.measure(1)
    mask, u, nbytes = lc.select(1e-3, 3)
    lc.pack_device(dst)
    lc.commit_snapshot()
    W, ou = _oracle_step(run, st, 1, 1e-3, 3)
    compare_decision(mask, u, run, ou, 1e-3)
    run.commit(run.last_mask, W)
    c0 = lc.counters()
    for t in range(2, 14):
        st.drift(t, scales)
        torch.cuda.synchronize()
        step = lc.step_graph_launch()
        assert step == t
        with pytest.raises(P.LCError):
            lc.step_graph_launch()        # the previous graph step must be read first
        mask, u, nbytes = lc.step_wait(t)
        W, ou = _oracle_step(run, st, t, 1e-3, 3)
        compare_decision(mask, u, run, ou, 1e-3)
        M, V = st.host_all("m"), st.host_all("v")
        stream_bytes, _ = run.pack(run.last_mask, W, M, V, t)
        run.commit(run.last_mask, W)
        torch.cuda.synchronize()
        got = (dst[:nbytes].cpu() if where == "device" else dst[:nbytes]).numpy()
        assert np.array_equal(got, stream_bytes), "graph step %d" % t
        for k in range(len(spec.tensors)):
            assert np.array_equal(st.host("R", k), run.R[k])
    assert lc.counters()["kernel_launches"] - c0["kernel_launches"] == 3 * 12
    lc.close()
