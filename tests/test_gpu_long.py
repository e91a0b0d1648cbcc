"""Long runs at the full sizes (slow).

* Llama-3-8B layout, 100 steps, tau in {5e-4, 1e-3, 2e-3}, S_max 8.  The
  oracle measures sampled layers in full at steps 1, 2, 50 and 100 and
  compares their packed blocks byte for byte; on every step the selection
  rule is re-checked on the CPU from the device's u (a select-only check)
  together with the staleness statistics.
* The cadence workload's drift regimes (uniform, top-heavy, bottom-heavy,
  sparse; switching every 50 steps) for 200 steps on the first 8
  transformer blocks of the 8B layout, persisted through a pinned ring
  store; at steps 50, 100 and 200 the run fails over: lc_restore writes
  the composite and the device state is compared with the oracle's
  composite bit for bit, then the run continues from it.
"""
import numpy as np
import pytest

from lc_workloads import gen, shapes
from lc_workloads.configs import WORKLOADS, cadence_scales
from oracle import oracle as O
from oracle.sim import OracleRun
from tests.lc_harness import U_RTOL, make_lc, oracle_measure_parallel, rel_err, require_gpu

pytestmark = [pytest.mark.gpu, pytest.mark.slow]


@pytest.mark.parametrize("tau", [5e-4, 1e-3, 2e-3])
def test_llama8b_100_steps(tau):
    torch = require_gpu()
    wl = WORKLOADS["8b"]
    spec = wl.shape()
    st = gen.SyntheticState(spec, device="cuda", seed=wl.seed)
    scales = wl.layer_scales(spec)
    K = wl.max_staleness
    lc = make_lc(st)
    run = OracleRun(st.tensor_layer, st.numels, st.nlayers, st.dtypes, st.has_moments,
                    keep_blocks="latest")
    sizes = np.array([sum(st.numels[k] for k in run.layer_tensors[l]) for l in range(spec.nlayers)])
    sample = [1, 16, 33]
    for l in sample:
        for k in run.layer_tensors[l]:
            run.R[k] = st.host("R", k)
    full = sum(lc.layer_block_bytes(l) for l in range(spec.nlayers))
    dst = torch.empty(full, dtype=torch.uint8, device="cuda")
    fractions = []
    for t in range(1, 101):
        st.drift(t, scales, redraw_moments=t in (1, 2, 50, 100))
        lc.measure(t)
        mask, u, nbytes = lc.select(tau, K)
        if t in (1, 2, 50, 100):
            ou, _ = oracle_measure_parallel(run, {k: st.host("W", k) for l in sample
                                                  for k in run.layer_tensors[l]}, layers=sample)
            err = rel_err(u[sample], ou[sample])
            assert err.max() <= U_RTOL, (t, dict(zip(sample, err)))
        omask, _, _ = O.select_step(u, run.delta, run.t_last, tau, K, t)
        assert np.array_equal(mask, omask), "select-only check at step %d" % t
        info = lc.info()
        mx, wt = O.staleness(run.t_last, sizes, t)
        assert info["max_staleness"] == mx <= K - 1 and info["weighted_staleness"] == wt
        fractions.append(mask.mean())
        lc.pack_device(dst)
        lc.commit_snapshot()
        if t in (1, 2, 50, 100):
            torch.cuda.synchronize()
            off = lc.offsets()
            for l in sample:
                if not mask[l]:
                    continue
                ts = [O.Tensor(st.host("W", k), None, st.host("m", k), st.host("v", k))
                      for k in run.layer_tensors[l]]
                block = O.pack_layer(ts, run.align)
                got = dst[int(off[l]):int(off[l]) + block.size].cpu().numpy()
                assert np.array_equal(got, block), "block of layer %d at step %d" % (l, t)
        for l in sample:
            if mask[l]:
                for k in run.layer_tensors[l]:
                    run.R[k] = st.host("W", k)
    assert 0.0 < np.mean(fractions) < 1.0
    lc.close()
    del st, dst
    torch.cuda.empty_cache()


def test_cadence_regimes_with_failovers():
    torch = require_gpu()
    import paper_2609_27193_gb300 as P
    wl = WORKLOADS["8b-cadence"]
    shape, _ = shapes.first_blocks(wl.shape(), 8)
    st = gen.SyntheticState(shape, device="cuda", seed=wl.seed)
    K, tau = wl.max_staleness, wl.tau
    lc = make_lc(st)
    run = OracleRun(st.tensor_layer, st.numels, st.nlayers, st.dtypes, st.has_moments,
                    keep_blocks="latest")
    store = P.Store(lc, versions_per_layer=2)
    checks = (50, 100, 200)
    windows = {t for c in checks for t in range(c - K + 1, c + 1)}

    def persist(mask, t):
        if t == 0 or t in windows:
            ks = [k for l in np.flatnonzero(mask) for k in run.layer_tensors[l]]
            W = {k: st.host("W", k) for k in ks}
            M = {k: st.host("m", k) for k in ks}
            V = {k: st.host("v", k) for k in ks}
            run.pack(mask, W, M, V, t)
            del W, M, V
        else:
            run.record(mask, t)
        lc.pack_async(store)
        lc.commit_snapshot()
        lc.wait_durable(t)
        run.mark_durable(t)

    lc.measure(0)
    mask, u, _ = lc.select(tau, 0)
    assert mask.all()
    O.select_step(u, run.delta, run.t_last, tau, 0, 0)
    persist(mask, 0)
    regimes = set()
    for t in range(1, 201):
        scales, regime = cadence_scales(wl, shape, t)
        regimes.add(regime)
        st.drift(t, scales)
        lc.measure(t)
        mask, u, nbytes = lc.select(tau, K)
        omask, _, _ = O.select_step(u, run.delta, run.t_last, tau, K, t)
        assert np.array_equal(mask, omask), "select-only check at step %d (%s)" % (t, regime)
        persist(mask, t)
        if t in checks:
            steps = lc.restore(store, t)
            comp, pick = run.composite(t)
            assert steps.tolist() == [run.versions[p]["step"] for p in pick]
            assert min(steps) >= t - K + 1
            torch.cuda.synchronize()
            for k in range(len(shape.tensors)):
                w, m, v = comp[k]
                assert np.array_equal(st.host("W", k), w), "W of tensor %d at %d" % (k, t)
                assert np.array_equal(st.host("R", k), w), "R of tensor %d at %d" % (k, t)
                assert np.array_equal(st.host("m", k), m), "m of tensor %d at %d" % (k, t)
                assert np.array_equal(st.host("v", k), v), "v of tensor %d at %d" % (k, t)
            del comp
            # after a recovery each layer carries its version's step and no drift
            run.t_last[:] = steps
            run.delta[:] = 0.0
            st.resync_master()
    assert regimes == set(wl.regimes)
    store.close()
    lc.close()
