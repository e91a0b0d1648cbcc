"""The ETTR model of §4.5 (Eq. 13-15): the event-driven failure simulation
against the exact expectation of the same process, limits, and the
checkpoint-interval optimum.  CPU only."""
import math

import pytest

from paper_2609_27193_gb300 import ettr as E


def test_no_failures_is_the_checkpoint_overhead():
    p = E.Policy("x", t_iter=2.0, k=1, t_ckpt_segment=0.5, t_load=10.0)
    assert E.expected_ettr(p, math.inf) == 2.0 / 2.5
    t = E.simulate(p, math.inf, 1000)
    assert t.failures == 0 and t.ettr == pytest.approx(0.8, rel=1e-12)


def test_free_checkpoints_lose_only_partial_iterations():
    # R = 0, no checkpoint cost: ETTR = lam*S / (e^{lam S} - 1)
    p = E.Policy("x", t_iter=3.0, k=1, t_ckpt_segment=0.0, t_load=0.0)
    mtbf = 60.0
    lam_s = 3.0 / mtbf
    assert E.expected_ettr(p, mtbf) == pytest.approx(lam_s / math.expm1(lam_s), rel=1e-12)


@pytest.mark.parametrize("k,ckpt,load,mtbf", [(1, 0.2, 5.0, 120.0), (10, 3.0, 20.0, 300.0),
                                              (1, 0.05, 1.0, 30.0), (40, 8.0, 60.0, 3600.0)])
def test_simulation_matches_exact_expectation(k, ckpt, load, mtbf):
    p = E.Policy("x", t_iter=1.5, k=k, t_ckpt_segment=ckpt, t_load=load, t_reconstruct=0.5, t_restart=2.0)
    want = E.expected_ettr(p, mtbf)
    iters = 200_000 if k < 10 else 400_000
    runs = [E.simulate(p, mtbf, iters, seed=s) for s in range(4)]
    got = sum(r.train for r in runs) / sum(r.wall for r in runs)
    nfail = sum(r.failures for r in runs)
    assert nfail > 400
    assert got == pytest.approx(want, rel=0.02)
    for r in runs:           # Eq. 13-15: the components add up to the wall time
        assert r.wall == pytest.approx(r.train + r.ckpt + r.load + r.reconstruct + r.restart + r.retrain)
        assert r.load == pytest.approx(r.failures * p.t_load)


def test_young_daly_interval_is_near_optimal():
    t_iter, c, mtbf, load = 2.0, 20.0, 3600.0, 30.0
    k_yd = E.young_daly_k(t_iter, c, mtbf)
    best = max(E.expected_ettr(E.Policy("p", t_iter, k, c, load), mtbf) for k in range(1, 2000))
    got = E.expected_ettr(E.Policy("p", t_iter, k_yd, c, load), mtbf)
    assert got >= 0.99 * best


def test_cheaper_checkpoints_and_rarer_failures_help():
    a = E.Policy("cheap", 2.0, 1, 0.05, 10.0)
    b = E.Policy("costly", 2.0, 1, 0.5, 10.0)
    for mtbf in (60.0, 600.0, 6000.0):
        assert E.expected_ettr(a, mtbf) > E.expected_ettr(b, mtbf)
    vals = [E.expected_ettr(a, m) for m in (60.0, 600.0, 6000.0, math.inf)]
    assert vals == sorted(vals)


def test_policies_from_a_bench_line():
    line = {"persisted_bytes_per_step": 20e9, "selected_fraction": 0.25, "ms_per_step": 12.0,
            "e2e": {"d2h_link_GBps_measured": 200.0}}
    pol = E.policies_from_bench(line, t_iter=2.0, h2d_gbps=200.0)
    assert pol["full_d2h"] == pytest.approx(80e9 / 200e9)
    assert pol["load"] == pytest.approx(0.4)
    assert pol["layercheck"].t_ckpt_segment == pytest.approx(0.012)     # D2H (0.1 s) hidden
    slow = E.policies_from_bench(line, t_iter=0.05, h2d_gbps=200.0)
    assert slow["layercheck"].t_ckpt_segment == pytest.approx(0.012 + 0.1 - 0.05)
    # a reported full-state size takes precedence over the layer-share estimate
    sized = E.policies_from_bench(dict(line, full_state_bytes=60e9), t_iter=2.0, h2d_gbps=200.0)
    assert sized["full_d2h"] == pytest.approx(60e9 / 200e9)
    assert sized["load"] == pytest.approx(0.3)
