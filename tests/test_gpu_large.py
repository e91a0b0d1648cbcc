"""GPU parity at the full workload sizes.

* Llama-3.2-1B shape, 50 steps (tau 1e-3, S_max 8) with the oracle in
  lockstep on every step: masks, measures, packed bytes (sampled steps) and
  the final composite restore.
* Llama-3-8B shape (35 layers) and its 291-tensor variant, in the launch
  configuration the benchmark times: the oracle computes the measures of
  sampled layers; the selection rule is re-checked on every layer from the
  device measures (a select-only check); sampled persisted blocks are
  compared byte for byte.
"""
import numpy as np
import pytest

from lc_workloads import gen, shapes
from lc_workloads.configs import WORKLOADS
from oracle import oracle as O
from oracle.sim import digest
from tests.lc_harness import (U_RTOL, compare_decision, make_lc, make_oracle,
                              oracle_measure_parallel, rel_err, require_gpu)

pytestmark = [pytest.mark.gpu, pytest.mark.slow]


def test_llama1b_50_steps_lockstep_and_restore():
    torch = require_gpu()
    import paper_2609_27193_gb300 as P
    wl = WORKLOADS["1b"]
    spec = wl.shape()
    st = gen.SyntheticState(spec, device="cuda", seed=wl.seed)
    scales = wl.layer_scales(spec)
    lc = make_lc(st)
    run = make_oracle(st, keep_blocks="latest")
    store = P.Store(lc, versions_per_layer=2)
    lc.measure(0)
    mask, _, nbytes = lc.select(wl.tau, 0)
    assert mask.all()
    W, M, V = st.host_all("W"), st.host_all("m"), st.host_all("v")
    run.select(np.zeros(spec.nlayers), wl.tau, 0, 0)
    run.pack(mask, W, M, V, 0)
    lc.pack_async(store)
    lc.commit_snapshot()
    lc.wait_durable(0)
    run.mark_durable(0)
    fractions = []
    for t in range(1, wl.steps + 1):
        st.drift(t, scales)
        W = st.host_all("W")
        lc.measure(t)
        mask, u, nbytes = lc.select(wl.tau, wl.max_staleness)
        ou, _ = oracle_measure_parallel(run, W)
        run.select(ou, wl.tau, wl.max_staleness, t)
        compare_decision(mask, u, run, ou, wl.tau)
        fractions.append(mask.mean())
        ks = [k for l in np.flatnonzero(run.last_mask) for k in run.layer_tensors[l]]
        M = {k: st.host("m", k) for k in ks}
        V = {k: st.host("v", k) for k in ks}
        stream, _ = run.pack(run.last_mask, W, M, V, t)
        assert nbytes == stream.size
        lc.pack_async(store)
        lc.commit_snapshot()
        run.commit(run.last_mask, W)
        lc.wait_durable(t)
        run.mark_durable(t)
        if t % 10 == 0:
            odig = {(v["layer"], v["step"]): v["digest"] for v in run.versions}
            for i, v in enumerate(store.versions()):
                if v["step"] == t:
                    assert digest(store.block(i)) == odig[(v["layer"], t)]
        del stream, M, V
    assert 0.1 < np.mean(fractions) < 0.6, "realized selection fraction %.3f" % np.mean(fractions)
    steps = lc.restore(store, wl.steps)
    comp, pick = run.composite(wl.steps)
    assert steps.tolist() == [run.versions[p]["step"] for p in pick]
    torch.cuda.synchronize()
    for k in range(len(spec.tensors)):
        w, m, v = comp[k]
        assert np.array_equal(st.host("W", k), w)
        assert np.array_equal(st.host("R", k), w)
        assert np.array_equal(st.host("m", k), m)
        assert np.array_equal(st.host("v", k), v)
    store.close()
    lc.close()


def _sampled_block_check(lc, st, run, mask, dst, sample_layers):
    off = lc.offsets()
    W = {}
    for l in sample_layers:
        if not mask[l]:
            continue
        for k in run.layer_tensors[l]:
            W[k] = st.host("W", k)
        ts = [O.Tensor(st.host("W", k), None, st.host("m", k), st.host("v", k))
              for k in run.layer_tensors[l]]
        block = O.pack_layer(ts, run.align)
        got = dst[int(off[l]):int(off[l]) + block.size].cpu().numpy()
        assert np.array_equal(got, block), "packed block of layer %d" % l


@pytest.mark.parametrize("per_tensor", [False, True])
def test_llama8b_sampled_parity(per_tensor):
    torch = require_gpu()
    wl = WORKLOADS["8b-tensor" if per_tensor else "8b"]
    spec = wl.shape()
    st = gen.SyntheticState(spec, device="cuda", seed=wl.seed)
    scales = wl.layer_scales(spec)
    lc = make_lc(st)
    from oracle.sim import OracleRun
    run = OracleRun(st.tensor_layer, st.numels, st.nlayers, st.dtypes, st.has_moments,
                    keep_blocks="latest")
    sizes = np.array([sum(st.numels[k] for k in run.layer_tensors[l]) for l in range(spec.nlayers)])
    if per_tensor:
        smallest = list(np.flatnonzero(sizes == sizes.min())[:2])
        sample = sorted(set(smallest + [0, 1, 4, 5, 289, 290, int(np.argmax(sizes))]))
    else:
        sample = [0, 1, 16, 33, 34]
    for l in sample:                 # the oracle keeps snapshots of the sampled layers only
        for k in run.layer_tensors[l]:
            run.R[k] = st.host("R", k)
    for t in (1, 2, 3):
        st.drift(t, scales, redraw_moments=(t == 3))
        lc.measure(t)
        mask, u, nbytes = lc.select(wl.tau, wl.max_staleness)
        # sampled layers: full oracle measure
        ou, _ = oracle_measure_parallel(run, {k: st.host("W", k) for l in sample
                                              for k in run.layer_tensors[l]}, layers=sample)
        err = rel_err(u[sample], ou[sample])
        assert err.max() <= U_RTOL, (t, dict(zip(sample, err)))
        # every layer: the selection rule re-checked on the device measures
        tl0, d0 = run.t_last.copy(), run.delta.copy()
        omask, _, _ = O.select_step(u, run.delta, run.t_last, wl.tau, wl.max_staleness, t)
        assert np.array_equal(mask, omask), "select-only check at step %d" % t
        info = lc.info()
        mx, wt = O.staleness(run.t_last, sizes, t)
        assert info["max_staleness"] == mx and info["weighted_staleness"] == wt
        dst = torch.empty(max(16, nbytes), dtype=torch.uint8, device="cuda")
        lc.pack_device(dst)
        lc.commit_snapshot()
        torch.cuda.synchronize()
        _sampled_block_check(lc, st, run, mask, dst, sample)
        # the oracle's own snapshot of the sampled layers follows the decisions;
        # the device snapshot of a persisted layer equals its weights
        for l in sample:
            for k in run.layer_tensors[l]:
                if mask[l]:
                    run.R[k] = st.host("W", k)
                assert np.array_equal(st.host("R", k), run.R[k])
        del dst
    lc.close()
    del st
    torch.cuda.empty_cache()
