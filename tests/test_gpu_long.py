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
* The same on the full 35-layer 8B layout with a bf16 matmul loop running
  on another stream throughout, through a newest-only store.
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


def _bits(t):
    """A tensor's raw bit pattern (so -0.0 and 0.0 differ)."""
    torch = require_gpu()
    return t.view(torch.int16) if t.element_size() == 2 else t.view(torch.int32)


def test_cadence_full_8b_layout_under_gemm_load():
    """The cadence workload at its full shape and load: the 35-layer
    Llama-3-8B layout (1.05 GB embed and lm_head weights) for 200 steps with
    the drift regimes switching every 50 steps, a bf16 8192^3 matmul loop on
    another stream all along, and the library on a side stream persisting
    through a newest-only pinned store.  On every step the selection rule is
    re-checked on the CPU from the device's u (select-only).  At steps 50,
    100 and 200 the run fails over: lc_restore writes the composite of §3.5 /
    Eq. 8 (under the matmul load as well), and

    * the chosen steps equal the oracle's pick over the durable versions;
    * every tensor's W, R, exp_avg and exp_avg_sq equal, bit for bit, the
      state captured when the oracle's picked version was persisted;
    * for the embedding, a middle block and lm_head the store's block equals
      the oracle's packed block of that state (§3.1) byte for byte, and the
      restored tensors equal the oracle's unpacked composite;

    then the run continues from the composite."""
    torch = require_gpu()
    import paper_2609_27193_gb300 as P
    wl = WORKLOADS["8b-cadence"]
    shape = wl.shape()
    N = shape.nlayers
    st = gen.SyntheticState(shape, device="cuda", seed=wl.seed)
    K, tau = wl.max_staleness, wl.tau
    main = torch.cuda.current_stream()
    side = torch.cuda.Stream()
    lc = make_lc(st, stream=side)
    run = OracleRun(st.tensor_layer, st.numels, st.nlayers, st.dtypes, st.has_moments, keep_blocks="latest")
    layer_tensors = run.layer_tensors
    blocks = [lc.layer_block_bytes(l) for l in range(N)]
    full = sum(blocks)
    sizes = sorted({-(-b // 4096) * 4096 for b in blocks})
    store = P.Store(lc, capacity_bytes=full + 2 * sum(sizes) + (1 << 30), versions_per_layer=1)
    # the state of every layer as it was when last persisted
    EW = [torch.empty_like(w) for w in st.W]
    EM = [torch.empty_like(m) for m in st.m]
    EV = [torch.empty_like(v) for v in st.v]
    gs = torch.cuda.Stream()
    a = torch.randn(8192, 8192, device="cuda", dtype=torch.bfloat16)
    b = torch.randn(8192, 8192, device="cuda", dtype=torch.bfloat16)
    c = torch.empty_like(a)

    def gemm_burst(n=40):
        with torch.cuda.stream(gs):
            for _ in range(n):
                torch.matmul(a, b, out=c)

    def capture(mask):
        for l in np.flatnonzero(mask):
            for k in layer_tensors[l]:
                EW[k].copy_(st.W[k])
                EM[k].copy_(st.m[k])
                EV[k].copy_(st.v[k])

    def persist(mask, t):
        capture(mask)
        lc.pack_async(store)
        lc.commit_snapshot()
        lc.wait_durable(t)
        run.record(mask, t)
        run.mark_durable(t)
        main.wait_stream(side)

    sample = [0, N // 2, N - 1]
    side.wait_stream(main)
    gemm_burst()
    lc.measure(0)
    mask, u, _ = lc.select(tau, 0)
    assert mask.all()
    O.select_step(u, run.delta, run.t_last, tau, 0, 0)
    persist(mask, 0)
    regimes, persisted = set(), []
    for t in range(1, 201):
        scales, regime = cadence_scales(wl, shape, t)
        regimes.add(regime)
        st.drift(t, scales)
        side.wait_stream(main)
        gemm_burst()
        lc.measure(t)
        mask, u, nbytes = lc.select(tau, K)
        omask, _, _ = O.select_step(u, run.delta, run.t_last, tau, K, t)
        assert np.array_equal(mask, omask), "select-only check at step %d (%s)" % (t, regime)
        persisted.append(nbytes)
        persist(mask, t)
        if t in (50, 100, 200):
            gemm_burst()
            steps = lc.restore(store, t)
            pick = run.pick(t)
            assert steps.tolist() == [run.versions[p]["step"] for p in pick], t
            assert min(steps) >= t - K + 1
            torch.cuda.synchronize()
            for k in range(len(shape.tensors)):
                for got, want, what in ((st.W[k], EW[k], "W"), (st.R[k], EW[k], "R"),
                                        (st.m[k], EM[k], "exp_avg"), (st.v[k], EV[k], "exp_avg_sq")):
                    assert torch.equal(_bits(got), _bits(want)), "%s of tensor %d at step %d" % (what, k, t)
            spick = store.plan(t)
            for l in sample:
                ts = [O.Tensor(gen.SyntheticState.to_numpy(EW[k]), None, gen.SyntheticState.to_numpy(EM[k]),
                               gen.SyntheticState.to_numpy(EV[k])) for k in layer_tensors[l]]
                block = O.pack_layer(ts, run.align)
                v = store.version(int(spick[l]))
                assert v["step"] == steps[l] and v["bytes"] == block.size
                assert np.array_equal(store.block(int(spick[l])), block), "block of layer %d at %d" % (l, t)
                shp = run._shape_tensors(l)
                O.unpack_layer(block, shp, run.align)
                for k, ex in zip(layer_tensors[l], shp):
                    assert np.array_equal(st.host("W", k), ex.w) and np.array_equal(st.host("R", k), ex.w)
                    assert np.array_equal(st.host("m", k), ex.m) and np.array_equal(st.host("v", k), ex.v)
                del ts, block, shp
            # after a recovery each layer carries its version's step and no drift
            run.t_last[:] = steps
            run.delta[:] = 0.0
            st.resync_master()
    assert regimes == set(wl.regimes)
    assert len(store) == N
    assert sum(persisted) > 0
    store.close()
    lc.close()
    del st, EW, EM, EV, a, b, c
    torch.cuda.empty_cache()


def test_llama8b_fused_adamw_sampled_parity():
    """The fused AdamW + drift step (§3.4.2) on the full Llama-3-8B layout in
    the launch configuration `bench.py --path fused` times: fp32 master
    weights as the optimizer's parameters, bf16 gradients and bf16 model
    copies, accumulate mode.  For sampled transformer blocks the updated
    weights, moments and model copies are bit-exact against the oracle's
    AdamW, and u within 1e-5; the selection rule is re-checked on every
    layer from the device's u, and sampled persisted blocks (fp32 weights
    and moments) are compared byte for byte."""
    torch = require_gpu()
    import paper_2609_27193_gb300 as P
    from lc_workloads.gen import mix_seed
    hp = (1e-5, 0.9, 0.999, 1e-8, 0.01)
    wl = WORKLOADS["8b"]
    spec = wl.shape()
    st = gen.SyntheticState(spec, device="cuda", seed=wl.seed, master=True, snapshot=False)
    lc = P.LayerCheck(mode=P.LC_DRIFT_ACCUMULATE)
    lc.register_layout([P.segment(t.layer, st.M[k], None, st.m[k], st.v[k])
                        for k, t in enumerate(spec.tensors)], spec.nlayers)
    grads = [torch.empty(t.numel, dtype=torch.bfloat16, device="cuda") for t in spec.tensors]
    lc.register_optimizer(grads, st.W)
    layer_tensors = [[k for k, t in enumerate(spec.tensors) if t.layer == l] for l in range(spec.nlayers)]
    sample = [1, 16, 33]
    delta = np.zeros(spec.nlayers)
    t_last = np.zeros(spec.nlayers, dtype=np.int64)
    tau, K = wl.tau, wl.max_staleness
    host = gen.SyntheticState.to_numpy
    for t in (1, 2):
        g = torch.Generator(device="cuda")
        for k, tsp in enumerate(spec.tensors):
            g.manual_seed(mix_seed(wl.seed, t, k, 5))
            grads[k].copy_(torch.randn(tsp.numel, generator=g, device="cuda").mul_(1e-3))
        torch.cuda.synchronize()
        ks = [k for l in sample for k in layer_tensors[l]]
        P0 = {k: host(st.M[k]) for k in ks}
        M0 = {k: host(st.m[k]) for k in ks}
        V0 = {k: host(st.v[k]) for k in ks}
        G = {k: host(grads[k]) for k in ks}
        lc.adamw_step_measure(t, hp[0], beta1=hp[1], beta2=hp[2], eps=hp[3], weight_decay=hp[4])
        mask, u, nbytes = lc.select(tau, K)
        torch.cuda.synchronize()
        for l in sample:
            d_l = a_l = n_l = 0.0
            for k in layer_tensors[l]:
                model = np.zeros(spec.tensors[k].numel, np.uint16)
                d, a = O.adamw_step(hp, t, P0[k], M0[k], V0[k], G[k], model)
                d_l, a_l, n_l = d_l + d, a_l + a, n_l + spec.tensors[k].numel
                assert np.array_equal(host(st.M[k]), P0[k]), "weights of tensor %d, step %d" % (k, t)
                assert np.array_equal(host(st.m[k]), M0[k]), "exp_avg of tensor %d" % k
                assert np.array_equal(host(st.v[k]), V0[k]), "exp_avg_sq of tensor %d" % k
                assert np.array_equal(host(st.W[k]), model), "model copy of tensor %d" % k
            ou = O.update_measure(d_l, a_l, n_l, 1e-8)
            assert rel_err(u[l:l + 1], np.array([ou]))[0] <= U_RTOL, (l, t, u[l], ou)
        omask, _, _ = O.select_step(u, delta, t_last, tau, K, t, O.ACCUMULATE)
        assert np.array_equal(mask, omask), "select-only check at step %d" % t
        dst = torch.empty(max(16, nbytes), dtype=torch.uint8, device="cuda")
        lc.pack_device(dst)
        lc.commit_snapshot()
        torch.cuda.synchronize()
        off = lc.offsets()
        for l in sample:
            if not mask[l]:
                continue
            ts = [O.Tensor(P0[k], None, M0[k], V0[k]) for k in layer_tensors[l]]
            block = O.pack_layer(ts)
            got = dst[int(off[l]):int(off[l]) + block.size].cpu().numpy()
            assert np.array_equal(got, block), "block of layer %d at step %d" % (l, t)
        del dst, P0, M0, V0, G
    lc.close()
    del st, grads
    torch.cuda.empty_cache()
