"""lc_measure_noalloc, the measure for callers that cannot allocate.

Some callers cannot call cudaMalloc once they run: a framework that owns
all GPU memory through its own pool, or a process whose device footprint is
fixed at start-up.  lc_measure_noalloc gives them the per-layer sums of
lc_measure without an lc_ctx; its scratch lives in a fixed-size static
device array.  These tests call it through the C ABI and compare its sums
with the oracle's, element by element within the tolerance of the measure
parity tests, on two calls in a row with different inputs (stale scratch
from the first call would show), with lc_measure's sums on the same tensors
in those two calls, on segments passed in shuffled layer order, and at
exactly LC_NOALLOC_MAX_SEGMENTS segments.  The file is named to be collected
last."""
import ctypes as C

import numpy as np
import pytest

from lc_workloads import gen, shapes
from lc_workloads.shapes import ModelShape, TensorSpec
from tests.lc_harness import U_RTOL, make_lc, make_oracle, oracle_measure_parallel, require_gpu

pytestmark = pytest.mark.gpu


def _segments(P, _abi, st, order):
    return (_abi.lc_segment * len(order))(*[P.segment(st.specs[k].layer, st.W[k], st.R[k])
                                            for k in order])


def _call(torch, lib, _abi, stream, segs, nseg, nlayers):
    out = torch.empty(3 * nlayers, dtype=torch.float64, device="cuda")
    with torch.cuda.stream(stream):
        out.fill_(float("nan"))
    _abi.check(lib.lc_measure_noalloc(0, C.c_void_p(stream.cuda_stream), segs, nseg, nlayers,
                                      C.c_void_p(out.data_ptr())))
    stream.synchronize()
    return out.cpu().numpy().reshape(-1, 3)


def _check_sums(got, want, what):
    assert np.all(np.isfinite(got)), "%s: a sum was not written" % what
    assert np.array_equal(got[:, 2], want[:, 2]), "%s: element counts differ" % what
    for col in (0, 1):
        den = np.maximum(np.abs(want[:, col]), 1e-300)
        rel = np.abs(got[:, col] - want[:, col]) / den
        assert rel.max() <= U_RTOL, (what, col, int(rel.argmax()), rel.max())


def _check_against_oracle(got, st, what):
    run = make_oracle(st)
    _, want = oracle_measure_parallel(run, st.host_all("W"))
    _check_sums(got, want, what)


def test_noalloc_measure_matches_oracle_on_two_calls():
    torch = require_gpu()
    import paper_2609_27193_gb300 as P
    from paper_2609_27193_gb300 import _abi
    lib = P.library()
    spec = shapes.tiny()
    # back-to-back views: odd-sized tensors make later ones start misaligned
    st = gen.SyntheticState(spec, device="cuda", seed=21, alloc="flat")
    n = len(spec.tensors)
    N = spec.nlayers
    # the tensors in a shuffled order: every layer's segments are interleaved
    order = list(np.random.default_rng(5).permutation(n))
    segs = _segments(P, _abi, st, order)
    stream = torch.cuda.Stream()
    scales = np.geomspace(1e-4, 3e-2, N)
    # the existing entry point on the same tensors, its sums in a buffer of ours
    lc = make_lc(st)
    ref = torch.zeros(3 * N, dtype=torch.float64, device="cuda")
    lc.set_layer_sums_buffer(ref)
    previous = None
    for t in (1, 2):
        st.drift(t, scales)
        torch.cuda.synchronize()
        got = _call(torch, lib, _abi, stream, segs, n, N)
        _check_against_oracle(got, st, "step %d" % t)
        lc.measure(t)
        lc.select(1e300, 1 << 30)          # persists nothing: R stays, the drift grows
        lc.commit_snapshot()
        torch.cuda.synchronize()
        _check_sums(got, ref.cpu().numpy().reshape(-1, 3), "lc_measure at step %d" % t)
        if previous is not None:
            assert not np.array_equal(previous[:, 0], got[:, 0]), "second call returned the first's sums"
        previous = got.copy()
    lc.close()


def test_noalloc_at_the_segment_limit():
    """Exactly LC_NOALLOC_MAX_SEGMENTS segments of uneven sizes and mixed
    dtypes over 40 layers, passed in shuffled order, then a small layout
    again on the same scratch."""
    torch = require_gpu()
    import paper_2609_27193_gb300 as P
    from paper_2609_27193_gb300 import _abi
    lib = P.library()
    rng = np.random.default_rng(11)
    nseg, nl = _abi.LC_NOALLOC_MAX_SEGMENTS, 40
    layers = np.concatenate([np.arange(nl), rng.integers(0, nl, nseg - nl)])
    sizes = rng.integers(1, 6000, nseg)
    sizes[::37] += 100000
    ts = [TensorSpec("t%d" % i, int(layers[i]), int(sizes[i]), "bf16" if i % 3 else "f32")
          for i in range(nseg)]
    spec = ModelShape("noalloc-limit", 0, 0, 0, 0, 0, 0, 0, False, False, ts, nl,
                      ["l%d" % i for i in range(nl)])
    st = gen.SyntheticState(spec, device="cuda", seed=4, alloc="flat", moments=False)
    st.drift(1, np.geomspace(1e-4, 1e-2, nl))
    torch.cuda.synchronize()
    order = list(rng.permutation(nseg))
    segs = _segments(P, _abi, st, order)
    stream = torch.cuda.Stream()
    got = _call(torch, lib, _abi, stream, segs, nseg, nl)
    _check_against_oracle(got, st, "512 segments")
    small = shapes.tiny()
    st2 = gen.SyntheticState(small, device="cuda", seed=8)
    st2.drift(1, np.full(small.nlayers, 3e-3))
    torch.cuda.synchronize()
    segs2 = _segments(P, _abi, st2, list(range(len(small.tensors))))
    got2 = _call(torch, lib, _abi, stream, segs2, len(small.tensors), small.nlayers)
    _check_against_oracle(got2, st2, "small layout after the large one")


def test_noalloc_rejects_bad_input_and_sizes_beyond_its_limits():
    torch = require_gpu()
    import paper_2609_27193_gb300 as P
    from paper_2609_27193_gb300 import _abi
    lib = P.library()
    w = torch.zeros(16, dtype=torch.bfloat16, device="cuda")
    r = torch.zeros(16, dtype=torch.bfloat16, device="cuda")
    out = torch.zeros(3 * 600, dtype=torch.float64, device="cuda")
    many = _abi.LC_NOALLOC_MAX_SEGMENTS + 1
    segs = (_abi.lc_segment * many)(*[P.segment(0, w, r) for _ in range(many)])
    st = lib.lc_measure_noalloc(0, None, segs, many, 1, C.c_void_p(out.data_ptr()))
    assert st == _abi.LC_ERR_CAPACITY
    assert b"LC_NOALLOC_MAX_SEGMENTS" in lib.lc_last_error()
    segs1 = (_abi.lc_segment * 1)(P.segment(0, w, r))
    st = lib.lc_measure_noalloc(0, None, segs1, 1, _abi.LC_NOALLOC_MAX_LAYERS + 1,
                                C.c_void_p(out.data_ptr()))
    assert st == _abi.LC_ERR_CAPACITY
    alias = (_abi.lc_segment * 1)(_abi.lc_segment(0, _abi.LC_BF16, w.data_ptr(), w.data_ptr(), None, None, 16))
    st = lib.lc_measure_noalloc(0, None, alias, 1, 1, C.c_void_p(out.data_ptr()))
    assert st == _abi.LC_ERR_INVALID_ARG
    assert b"alias" in lib.lc_last_error()
