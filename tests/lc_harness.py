"""Shared helpers of the GPU parity tests: run the CUDA path and the oracle
side by side on the same seeded inputs.

The CUDA path is reached only through the C ABI (the ctypes binding); the
oracle keeps its own reference copies, accumulators, last-persistence steps
and store, fed with host copies of the generator's inputs -- never with
anything the CUDA path computed.
"""
import concurrent.futures as cf
import os

import numpy as np
import pytest

U_RTOL = 1e-5      # per-layer measures: GPU fp32 partials vs the fp64 oracle


def require_gpu():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2609_27193_gb300 import build as B
    B.build()
    return torch


def make_lc(state, stream=None, tau_mult=None, **kw):
    import paper_2609_27193_gb300 as P
    lc = P.LayerCheck(device=state.device.index or 0, stream=stream, **kw)
    segs = [P.segment(state.specs[k].layer, state.W[k], state.R[k], state.m[k], state.v[k])
            for k in range(len(state.specs))]
    lc.register_layout(segs, state.nlayers, tau_mult)
    return lc


def make_oracle(state, keep_blocks="all", tau_mult=None, **kw):
    from oracle.sim import OracleRun
    run = OracleRun(state.tensor_layer, state.numels, state.nlayers, state.dtypes,
                    state.has_moments, keep_blocks=keep_blocks, tau_mult=tau_mult, **kw)
    run.set_reference(state.host_all("R"))
    return run


_POOL = None


def pool():
    global _POOL
    if _POOL is None:
        _POOL = cf.ThreadPoolExecutor(max_workers=max(1, min(16, os.cpu_count() or 1)))
    return _POOL


def oracle_measure_parallel(run, W, layers=None):
    """The oracle's per-layer sums, one layer per worker thread (the C oracle
    releases the GIL; each layer is still summed in its plain order)."""
    from oracle import oracle as O
    ls = list(range(run.nlayers)) if layers is None else list(layers)

    def one(l):
        d, a, n = O.layer_sums(run._tensors(l, W))
        return l, d, a, n

    u = np.full(run.nlayers, np.nan)
    sums = np.full((run.nlayers, 3), np.nan)
    for l, d, a, n in pool().map(one, ls):
        sums[l] = (d, a, n)
        u[l] = O.update_measure(d, a, n, run.eps_w)
    return u, sums


def rel_err(a, b):
    a = np.asarray(a, dtype=np.float64)
    b = np.asarray(b, dtype=np.float64)
    den = np.maximum(np.abs(b), 1e-300)
    return np.abs(a - b) / den


def compare_decision(gpu_mask, gpu_u, run, oracle_u, tau, tau_mult=None):
    """Checks u within U_RTOL and the masks; a layer whose accumulated drift
    lies within U_RTOL * tau of its threshold is flagged, and the oracle then
    takes the GPU's decision for it.  Returns the flagged layers."""
    finite = np.isfinite(oracle_u)
    assert np.array_equal(np.isfinite(gpu_u), finite), "finite pattern of u differs"
    if finite.any():
        err = rel_err(gpu_u[finite], oracle_u[finite])
        assert err.max() <= U_RTOL, "u differs by %.3g relative (layer %d)" % (
            err.max(), np.flatnonzero(finite)[err.argmax()])
    return adopt_flagged(gpu_mask, run, tau, tau_mult)


def adopt_flagged(gpu_mask, run, tau, tau_mult=None):
    from oracle import oracle as O
    acc_before, _, u, _ = run._undo
    acc = acc_before + u if run.mode == O.ACCUMULATE else u
    thr = tau * (np.ones(run.nlayers) if tau_mult is None else np.asarray(tau_mult))
    flagged = np.isfinite(acc) & (np.abs(acc - thr) <= U_RTOL * np.abs(thr))
    mask = run.last_mask
    mism = np.flatnonzero(gpu_mask != mask)
    bad = [l for l in mism if not flagged[l]]
    assert not bad, "selection differs on layers %s (not in the tolerance band)" % bad
    for l in mism:
        run.adopt_decision(int(l), bool(gpu_mask[l]))
        mask[l] = gpu_mask[l]
    return list(mism)
