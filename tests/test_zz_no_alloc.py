"""lc_measure_noalloc, the allocation-free form of the Eq. 1 measure.

Some callers cannot call cudaMalloc once they run: a framework that owns
all GPU memory through its own pool, or a process whose device footprint is
fixed at start-up.  lc_measure_noalloc gives them the per-layer sums
without creating a context; its scratch lives in a fixed-size static device
array.  This checks it through the C ABI against the context-based
lc_measure, on two calls in a row with different inputs (so stale scratch
from the first call would show), within the tolerance of the measure parity
tests.  The file is named to be collected last."""
import ctypes as C

import numpy as np
import pytest

from lc_workloads import gen, shapes
from tests.lc_harness import U_RTOL, make_lc, require_gpu

pytestmark = pytest.mark.gpu


def test_noalloc_measure_matches_lc_measure_on_two_calls():
    torch = require_gpu()
    import paper_2609_27193_gb300 as P
    from paper_2609_27193_gb300 import _abi
    lib = P.library()
    spec = shapes.tiny()
    # back-to-back views: odd-sized tensors make later ones start misaligned
    st = gen.SyntheticState(spec, device="cuda", seed=21, alloc="flat")
    n = len(spec.tensors)
    N = spec.nlayers
    segs = (_abi.lc_segment * n)(*[P.segment(t.layer, st.W[k], st.R[k], st.m[k], st.v[k])
                                   for k, t in enumerate(spec.tensors)])
    stream = torch.cuda.Stream()
    lc = make_lc(st, stream=stream)
    ref = torch.zeros(3 * N, dtype=torch.float64, device="cuda")
    lc.set_layer_sums_buffer(ref)
    out = torch.empty(3 * N, dtype=torch.float64, device="cuda")
    scales = np.geomspace(1e-4, 3e-2, N)
    previous = None
    for t in (1, 2):
        st.drift(t, scales)
        torch.cuda.synchronize()
        lc.measure(t)
        lc.select(1e30, 1000)            # closes the step; nothing persists, R is unchanged
        with torch.cuda.stream(stream):
            out.fill_(float("nan"))
        _abi.check(lib.lc_measure_noalloc(0, C.c_void_p(stream.cuda_stream), segs, n, N,
                                          C.c_void_p(out.data_ptr())))
        stream.synchronize()
        got = out.cpu().numpy().reshape(-1, 3)
        want = ref.cpu().numpy().reshape(-1, 3)
        assert np.all(np.isfinite(got)), "a sum was not written"
        assert np.array_equal(got[:, 2], want[:, 2]), "element counts differ"
        for col in (0, 1):
            rel = np.abs(got[:, col] - want[:, col]) / np.abs(want[:, col])
            assert rel.max() <= U_RTOL, (t, col, rel.max())
        if previous is not None:
            assert not np.array_equal(previous[:, 0], got[:, 0]), "second call returned the first's sums"
        previous = got.copy()
    lc.close()


def test_noalloc_rejects_sizes_beyond_its_limits():
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
