"""GPU parity of the measure (Eq. 1) and select (Eq. 2-4, §3.3) kernels
against the oracle, through the C ABI."""
import math
import os

import numpy as np
import pytest

from lc_workloads import gen, shapes
from lc_workloads.shapes import ModelShape, TensorSpec
from oracle import oracle as O
from tests.conftest import GOLDEN
from tests.lc_harness import (U_RTOL, compare_decision, make_lc, make_oracle, oracle_measure_parallel,
                              rel_err, require_gpu)

pytestmark = pytest.mark.gpu


def custom_shape(sizes_layers, name="custom"):
    """sizes_layers: list of (numel, layer)."""
    ts = [TensorSpec("t%d" % i, l, n) for i, (n, l) in enumerate(sizes_layers)]
    nl = max(l for _, l in sizes_layers) + 1
    return ModelShape(name, 0, 0, 0, 0, 0, 0, 0, False, False, ts, nl, ["l%d" % i for i in range(nl)])


def _bf16_vals(vals):
    return np.asarray(vals, dtype=np.float32)


# ----------------------------------------------------------------------------
# hand cases: exact sums, so u is bit-exact
# ----------------------------------------------------------------------------

@pytest.mark.parametrize("engine", ["bulk", "threads"])
def test_hand_cases_exact(engine):
    torch = require_gpu()
    eps = 1e-8
    # H1 layer A, H1 layer B, H3 (two tensors), H2
    spec = custom_shape([(2, 0), (2, 1), (1, 2), (3, 2), (2, 3)])
    st = gen.SyntheticState(spec, device="cuda", seed=0)
    vals = {0: ([1, 2], [1, 2]), 1: ([1.5, -1], [1, -1]), 2: ([2], [1]), 3: ([1, 1, 1], [1, 1, 1]),
            4: ([0, 2.0 ** -10], [0, 0])}
    for k, (w, r) in vals.items():
        st.set_values(k, w=_bf16_vals(w), r=_bf16_vals(r))
    lc = make_lc(st, eps_w=eps, copy_engine=engine)
    sums = torch.zeros(3 * spec.nlayers, dtype=torch.float64, device="cuda")
    lc.set_layer_sums_buffer(sums)
    lc.measure(1)
    mask, u, nbytes = lc.select(0.25, 100)
    s = sums.cpu().numpy().reshape(-1, 3)
    assert s[0].tolist() == [0.0, 3.0, 2.0]
    assert s[1].tolist() == [0.5, 2.0, 2.0]
    assert s[2].tolist() == [1.0, 4.0, 4.0]
    assert s[3].tolist() == [2.0 ** -10, 0.0, 2.0]
    assert u[0] == 0.0
    assert u[1] == 0.25 / (1 + eps)
    assert u[2] == 0.25 / (1 + eps)
    assert u[3] == 2.0 ** -11 / eps
    # tau = 0.25 sits just above 0.25/(1+eps): only H2 persists
    assert mask.tolist() == [0, 0, 0, 1]
    assert lc.counters()["bulk_measure_launches"] == (1 if engine == "bulk" else 0)
    lc.close()


# ----------------------------------------------------------------------------
# edge shapes, dtypes and alignments vs the oracle
# ----------------------------------------------------------------------------

EDGE_SIZES = [1, 7, 8, 9, 4095, 4096, (1 << 20) + 3, 33, 2, 100003]


@pytest.mark.parametrize("engine", ["bulk", "threads"])
@pytest.mark.parametrize("alloc", ["separate", "flat", "skew"])
@pytest.mark.parametrize("dtype", ["bf16", "f32", "mixed"])
def test_measure_edge_shapes(alloc, dtype, engine):
    require_gpu()
    sizes = [(n, i % 4) for i, n in enumerate(EDGE_SIZES)]
    spec = custom_shape(sizes)
    if dtype == "mixed":
        dts = ["bf16" if i % 3 else "f32" for i in range(len(sizes))]
    else:
        dts = [dtype] * len(sizes)
    st = gen.SyntheticState(spec, device="cuda", seed=5, alloc=alloc, dtypes=dts)
    scales = np.array([3e-3, 1e-2, 1e-4, 5e-2])
    st.drift(1, scales)
    lc = make_lc(st, copy_engine=engine)
    run = make_oracle(st)
    lc.measure(1)
    mask, u, _ = lc.select(1e-3, 100)
    ou, _ = run.measure(st.host_all("W"))
    run.select(ou, 1e-3, 100, 1)
    compare_decision(mask, u, run, ou, 1e-3)
    lc.close()


@pytest.mark.parametrize("mode", ["snapshot", "accumulate"])
@pytest.mark.parametrize("alloc", ["flat", "skew"])
def test_measure_pool_of_ranges_with_odd_segments(alloc, mode):
    """The bulk measure's CTAs take small ranges from a pool once their own
    range is done; unit boundaries then fall anywhere in the work space.
    About 1.2 G elements in odd-sized segments of mixed dtypes over five
    layers, packed back to back (flat: most segments start off a 16-byte
    boundary, W and R alike) or with R shifted by one element (skew: W and R
    never co-aligned, so every run goes element by element): enough for the
    library to use a pool, and the sums must match the oracle's.  In
    accumulate mode (six consumer warps and a storer that writes R <- W) R
    must equal W afterwards, bit for bit, in every tensor."""
    torch = require_gpu()
    import paper_2609_27193_gb300 as P
    acc = mode == "accumulate"
    rng = np.random.default_rng(17)
    big = [int(x) | 1 for x in rng.integers(20_000_000, 140_000_000, size=14)]
    small = [1, 3, 7, 33, 4097, 65535, 1000003]
    sizes = [(n, i % 5) for i, n in enumerate(big[:7] + small + big[7:])]
    spec = custom_shape(sizes)
    dts = ["f32" if i % 4 == 1 else "bf16" for i in range(len(sizes))]
    st = gen.SyntheticState(spec, device="cuda", seed=23, alloc=alloc, dtypes=dts, master=False)
    st.drift(1, np.array([2e-2, 3e-3, 1e-2, 5e-2, 8e-3]))
    lc = make_lc(st, copy_engine="bulk", mode=P.LC_DRIFT_ACCUMULATE if acc else P.LC_DRIFT_SNAPSHOT)
    assert lc.counters()["measure_pool_units"] > 0, "layout too small for a pool"
    run = make_oracle(st, mode=O.ACCUMULATE if acc else O.SNAPSHOT)
    lc.measure(1)
    mask, u, _ = lc.select(1e-3, 100)
    ou, _ = oracle_measure_parallel(run, st.host_all("W"))
    run.select(ou, 1e-3, 100, 1)
    compare_decision(mask, u, run, ou, 1e-3)
    if acc:
        torch.cuda.synchronize()
        for k in range(len(spec.tensors)):
            bits = torch.int16 if st.W[k].element_size() == 2 else torch.int32
            assert torch.equal(st.R[k].view(bits), st.W[k].view(bits)), "R <- W of tensor %d" % k
    lc.close()


@pytest.mark.parametrize("engine", ["bulk", "threads"])
def test_measure_interleaved_registration_and_many_segments(engine):
    """Layer ids in any registration order; hundreds of uneven segments."""
    require_gpu()
    rng = np.random.default_rng(3)
    sizes = []
    for i in range(300):
        n = int(rng.choice([1, 5, 64, 4096, 12345, 70001]))
        sizes.append((n, int(rng.integers(0, 37))))
    for l in range(37):                      # every layer has a tensor
        sizes.append((17 + l, l))
    spec = custom_shape(sizes)
    st = gen.SyntheticState(spec, device="cuda", seed=8, alloc="flat")
    st.drift(1, gen.loguniform(37, 1e-4, 3e-2, rng))
    lc = make_lc(st, copy_engine=engine)
    run = make_oracle(st)
    lc.measure(1)
    mask, u, _ = lc.select(2e-3, 100)
    ou, _ = run.measure(st.host_all("W"))
    run.select(ou, 2e-3, 100, 1)
    compare_decision(mask, u, run, ou, 2e-3)
    lc.close()


@pytest.mark.parametrize("engine", ["bulk", "threads"])
def test_measure_deterministic_and_zero_drift(engine):
    torch = require_gpu()
    spec = shapes.tiny()
    st = gen.SyntheticState(spec, device="cuda", seed=1)
    lc = make_lc(st, copy_engine=engine)
    # W == R: every layer measures exactly 0 (Eq. 1 numerator)
    lc.measure(1)
    mask, u, _ = lc.select(1e-3, 100)
    assert np.all(u == 0.0) and mask.sum() == 0
    st.drift(2, np.full(spec.nlayers, 1e-3))
    us = []
    for t in (2, 3):
        lc.measure(t)
        _, u, _ = lc.select(1.0, 100)      # nothing persists: R stays the same
        us.append(u)
    assert np.array_equal(us[0], us[1]), "measure is not deterministic"
    lc.close()


def test_nonfinite_and_zero_reference_layers_persist():
    torch = require_gpu()
    spec = custom_shape([(1000, 0), (1000, 1), (1000, 2), (1000, 3)])
    st = gen.SyntheticState(spec, device="cuda", seed=2)
    with torch.no_grad():
        st.W[0][10] = float("nan")
        st.W[1][999] = float("inf")
        st.R[2].zero_()
        st.W[2].zero_()
        st.W[2][5] = 2.0 ** -10
    lc = make_lc(st)
    run = make_oracle(st)
    lc.measure(1)
    mask, u, _ = lc.select(1e-3, 100)
    info = lc.info()
    ou, _ = run.measure(st.host_all("W"))
    omask = run.select(ou, 1e-3, 100, 1)
    assert mask.tolist() == omask.tolist() == [1, 1, 1, 0]
    assert info["n_nonfinite"] == 2
    assert math.isnan(u[0]) and math.isinf(u[1]) and u[2] == ou[2]
    lc.close()


# ----------------------------------------------------------------------------
# select kernel: golden sequences and brute force, with injected measures
# ----------------------------------------------------------------------------

def _select_with_u(lc, sums, us, tau, K, t):
    """Runs the device select on given u values: with eps_w = 1, D = u,
    A = 0, n = 1 gives u exactly."""
    import torch
    lc.measure(t)
    inj = np.zeros((len(us), 3))
    inj[:, 0] = us
    inj[:, 2] = 1.0
    with torch.cuda.stream(lc.stream):
        sums.copy_(torch.from_numpy(inj.reshape(-1)).to("cuda", non_blocking=False))
    return lc.select(tau, K)


def _sequences():
    out = []
    with open(os.path.join(GOLDEN, "select_sequences.txt")) as fh:
        for line in fh:
            line = line.split("#", 1)[0].strip()
            if line:
                head, us, masks = [p.split() for p in line.split("|")]
                out.append((head[0], head[1], float(head[2]), int(head[3]),
                            [float(x) for x in us], [int(x) for x in masks]))
    return out


@pytest.mark.parametrize("mode", ["snapshot", "accumulate"])
def test_select_golden_sequences_on_device(mode):
    torch = require_gpu()
    import paper_2609_27193_gb300 as P
    seqs = [s for s in _sequences() if s[1] == mode]
    assert seqs
    for name, _, tau, K, us, want in seqs:
        spec = custom_shape([(16, 0)])
        st = gen.SyntheticState(spec, device="cuda", seed=0)
        lc = make_lc(st, eps_w=1.0,
                     mode=P.LC_DRIFT_ACCUMULATE if mode == "accumulate" else P.LC_DRIFT_SNAPSHOT)
        sums = torch.zeros(3, dtype=torch.float64, device="cuda")
        lc.set_layer_sums_buffer(sums)
        got = []
        for t, u in enumerate(us, start=1):
            mask, _, _ = _select_with_u(lc, sums, [u], tau, K, t)
            got.append(int(mask[0]))
            if mask[0]:
                lc.pack_device(torch.empty(lc.info()["bytes"], dtype=torch.uint8, device="cuda"))
            lc.commit_snapshot()
        assert got == want, name
        lc.close()


def test_select_brute_force_and_staleness_stats():
    """Every drift sequence of 3 layers over 4 steps from {0, tau/2, tau, 2tau}
    (sampled) and K in 0..4, both modes: masks, accumulators (via the next
    decisions) and the staleness statistics equal the oracle's bit for bit."""
    torch = require_gpu()
    import paper_2609_27193_gb300 as P
    rng = np.random.default_rng(0)
    tau = 0.5
    vals = np.array([0.0, tau / 2, tau, 2 * tau])
    numel = [3, 1000, 77]
    for mode in (O.SNAPSHOT, O.ACCUMULATE):
        for K in range(0, 5):
            spec = custom_shape([(n, l) for l, n in enumerate(numel)])
            st = gen.SyntheticState(spec, device="cuda", seed=0)
            lc = make_lc(st, eps_w=1.0, mode=mode)
            sums = torch.zeros(9, dtype=torch.float64, device="cuda")
            lc.set_layer_sums_buffer(sums)
            delta = np.zeros(3)
            tl = np.zeros(3, dtype=np.int64)
            for t in range(1, 41):
                us = rng.choice(vals, 3)
                mask, u, _ = _select_with_u(lc, sums, us, tau, K, t)
                omask, _, _ = O.select_step(us, delta, tl, tau, K, t, mode)
                assert mask.tolist() == omask.tolist(), (mode, K, t)
                info = lc.info()
                mx, wt = O.staleness(tl, numel, t)
                assert info["max_staleness"] == mx and info["weighted_staleness"] == wt
                if mask.any():
                    lc.pack_device(torch.empty(info["bytes"], dtype=torch.uint8, device="cuda"))
                lc.commit_snapshot()
            lc.close()


def test_tau_multiplier():
    torch = require_gpu()
    spec = custom_shape([(8, 0), (8, 1)])
    st = gen.SyntheticState(spec, device="cuda", seed=0)
    lc = make_lc(st, eps_w=1.0, tau_mult=[10.0, 1.0])
    sums = torch.zeros(6, dtype=torch.float64, device="cuda")
    lc.set_layer_sums_buffer(sums)
    mask, _, _ = _select_with_u(lc, sums, [5e-3, 5e-3], 1e-3, 100, 1)
    assert mask.tolist() == [0, 1]
    lc.close()


def test_api_errors_and_state_machine():
    torch = require_gpu()
    import paper_2609_27193_gb300 as P
    spec = custom_shape([(64, 0), (64, 1)])
    st = gen.SyntheticState(spec, device="cuda", seed=0)
    lc = P.LayerCheck(device=0)
    with pytest.raises(P.LCError) as e:
        lc.measure(1)
    assert e.value.status == 2
    # a layer without segments
    segs = [P.segment(0, st.W[0], st.R[0], st.m[0], st.v[0])]
    with pytest.raises(P.LCError) as e:
        lc.register_layout(segs, 2)
    assert e.value.status == 1
    # host memory is rejected
    hw = torch.zeros(64, dtype=torch.bfloat16)
    bad = [P.segment(0, hw, hw), P.segment(1, st.W[1], st.R[1])]
    with pytest.raises(P.LCError):
        lc.register_layout(bad, 2)
    lc.close()
    lc = make_lc(st)
    with pytest.raises(P.LCError) as e:
        lc.select(1e-3, 4)
    assert e.value.status == 2
    lc.measure(3)
    with pytest.raises(P.LCError):
        lc.select(float("nan"), 4)
    with pytest.raises(P.LCError):
        lc.select(1e-3, -1)
    mask, _, nbytes = lc.select(1e-3, 0)     # S_max = 0: everything persists
    assert mask.tolist() == [1, 1]
    with pytest.raises(P.LCError) as e:
        lc.measure(4)                          # step still open
    assert e.value.status == 2
    with pytest.raises(P.LCError) as e:
        lc.commit_snapshot()                   # not packed
    assert e.value.status == 2
    small = torch.empty(16, dtype=torch.uint8, device="cuda")
    with pytest.raises(P.LCError) as e:
        lc.pack_device(small)
    assert e.value.status == 5
    lc.pack_device(torch.empty(nbytes, dtype=torch.uint8, device="cuda"))
    lc.commit_snapshot()
    with pytest.raises(P.LCError):
        lc.measure(3)                          # steps must increase
    lc.measure(4)
    lc.select(1e-3, 100)
    lc.close()


def test_bulk_measure_wait_bound_reports_timeout():
    """LC_DEBUG_MEASURE_STALL: each CTA of the bulk-load measure waits for 16
    bytes that never arrive; the waits give up after 1 s, the kernel returns,
    and lc_select fails with LC_ERR_TIMEOUT instead of taking a decision
    from incomplete sums.  A fresh context on the same device still works."""
    import time
    torch = require_gpu()
    import paper_2609_27193_gb300 as P
    spec = shapes.tiny()
    st = gen.SyntheticState(spec, device="cuda", seed=2)
    st.drift(1, np.full(spec.nlayers, 1e-2))
    lc = make_lc(st, debug_flags=P.LC_DEBUG_MEASURE_STALL)
    t0 = time.perf_counter()
    lc.measure(1)
    with pytest.raises(P.LCError) as e:
        lc.select(1e-3, 100)
    assert e.value.status == 6
    assert time.perf_counter() - t0 < 30.0
    assert lc.counters()["bulk_measure_launches"] == 1
    lc.close()
    lc2 = make_lc(st)
    run = make_oracle(st)
    lc2.measure(1)
    mask, u, _ = lc2.select(1e-3, 100)
    ou, _ = run.measure(st.host_all("W"))
    run.select(ou, 1e-3, 100, 1)
    compare_decision(mask, u, run, ou, 1e-3)
    lc2.close()
