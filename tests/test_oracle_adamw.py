"""Pins of the oracle's fused AdamW + drift step (§3.4.2: the drift of
Eq. 1 is read off the optimizer update) against hand-worked values, closed
forms, an independent binary64 AdamW, and torch's bf16 rounding."""
import math
import os

import numpy as np
import pytest

from oracle import oracle as O
from tests.conftest import GOLDEN


def _cases():
    out = []
    for line in open(os.path.join(GOLDEN, "adamw_hand_cases.txt")):
        line = line.split("#", 1)[0].strip()
        if not line:
            continue
        head, ins, outs, sums = [p.strip() for p in line.split("|")]
        h = head.split()
        name, t, hp = h[0], int(h[1]), tuple(float(x) for x in h[2:7])
        ins = [[float(x) for x in e.split()] for e in ins.split(";")]
        outs = [[float(x) for x in e.split()] for e in outs.split(";")]
        out.append((name, t, hp, ins, outs, [float(x) for x in sums.split()]))
    return out


def test_adamw_hand_cases(oracle_lib):
    cases = _cases()
    assert len(cases) == 4
    for name, t, hp, ins, outs, (d_exp, a_exp) in cases:
        p = np.array([e[0] for e in ins], np.float32)
        m = np.array([e[1] for e in ins], np.float32)
        v = np.array([e[2] for e in ins], np.float32)
        g = np.array([e[3] for e in ins], np.float32)
        d, a = O.adamw_step(hp, t, p, m, v, g)
        assert p.tolist() == [e[0] for e in outs], name
        assert m.tolist() == [e[1] for e in outs], name
        assert v.tolist() == [e[2] for e in outs], name
        assert (d, a) == (d_exp, a_exp), name


def test_constant_gradient_closed_form(oracle_lib):
    # With beta = 1/2 and g = 1, m_t = 1 - 2^-t = 1 - beta1^t exactly, so the
    # bias-corrected m_hat = v_hat = 1 and p drops by exactly lr each step.
    p = np.array([1.0, -3.0], np.float32)
    m = np.zeros(2, np.float32)
    v = np.zeros(2, np.float32)
    g = np.array([1.0, 1.0], np.float32)
    for t in range(1, 21):
        O.adamw_step((2.0 ** -6, 0.5, 0.5, 0.0, 0.0), t, p, m, v, g)
        assert p.tolist() == [1.0 - t * 2.0 ** -6, -3.0 - t * 2.0 ** -6]


def _adamw64(hp, t, p, m, v, g):
    lr, b1, b2, eps, wd = hp
    p = p.astype(np.float64) * (1.0 - lr * wd)
    m = b1 * m.astype(np.float64) + (1.0 - b1) * g
    v = b2 * v.astype(np.float64) + (1.0 - b2) * g * g
    mh = m / (1.0 - b1 ** t)
    vh = v / (1.0 - b2 ** t)
    return p - lr * mh / (np.sqrt(vh) + eps), m, v


def test_matches_binary64_adamw_within_fp32_rounding(oracle_lib):
    rng = np.random.default_rng(0)
    n = 20000
    hp = (1e-3, 0.9, 0.999, 1e-8, 0.01)
    p = (rng.standard_normal(n) * 0.02).astype(np.float32)
    m = (rng.standard_normal(n) * 1e-3).astype(np.float32)
    v = np.abs(rng.standard_normal(n) * 1e-6).astype(np.float32)
    g = (rng.standard_normal(n) * 1e-2).astype(np.float32)
    for t in (1, 7, 100):
        p64, m64, v64 = _adamw64(hp, t, p, m, v, g.astype(np.float64))
        pp, mm, vv = p.copy(), m.copy(), v.copy()
        O.adamw_step(hp, t, pp, mm, vv, g)
        # each fp32 operation rounds once (relative 2^-24) and the constants
        # are fp32 roundings of the binary64 hyperparameters; errors are
        # bounded relative to the operands, which can cancel
        u = 2.0 ** -24
        lr, b1, b2, eps, wd = hp
        m_terms = np.abs(b1 * m.astype(np.float64)) + np.abs((1 - b1) * g.astype(np.float64))
        step = np.abs(p64 - p.astype(np.float64) * (1 - lr * wd))
        p_terms = np.abs(p.astype(np.float64) * (1 - lr * wd))
        assert np.all(np.abs(mm - m64) <= 4 * u * m_terms), t
        assert np.all(np.abs(vv - v64) <= 4 * u * np.abs(v64)), t
        assert np.all(np.abs(pp - p64) <= 4 * u * p_terms + 16 * u * step), t
        # and a dropped bias correction or weight decay would be far outside
        assert np.abs(pp - p64).max() < 1e-3 * step.max()


def test_fused_drift_sums_are_eq1_of_the_update(oracle_lib):
    rng = np.random.default_rng(1)
    n = 5001
    hp = (3e-4, 0.9, 0.95, 1e-8, 0.1)
    p = (rng.standard_normal(n) * 0.02).astype(np.float32)
    m = (rng.standard_normal(n) * 1e-3).astype(np.float32)
    v = np.abs(rng.standard_normal(n) * 1e-6).astype(np.float32)
    gbits = ((rng.standard_normal(n) * 1e-2).astype(np.float32).view(np.uint32) >> 16).astype(np.uint16)
    p_old = p.copy()
    model = np.zeros(n, np.uint16)
    d, a = O.adamw_step(hp, 3, p, m, v, gbits, model)
    d2, a2, cnt = O.layer_sums([O.Tensor(p, p_old)])
    assert (d, a) == (d2, a2) and cnt == n
    assert d > 0
    # the model copy is bf16(p_new), nearest even
    assert all(model[i] == O.bf16_round(p[i]) for i in range(0, n, 97))


def test_bf16_round_matches_torch():
    torch = pytest.importorskip("torch")
    rng = np.random.default_rng(2)
    f = np.concatenate([rng.standard_normal(3000).astype(np.float32) * s for s in (1e-3, 1, 1e4)])
    ties = ((np.arange(256, dtype=np.uint32) << 16) | 0x8000).view(np.float32)   # exactly half way
    f = np.concatenate([f, ties, np.array([0.0, -0.0, np.inf, -np.inf, 3.4e38], np.float32)])
    want = torch.from_numpy(f).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    got = np.array([O.bf16_round(x) for x in f], dtype=np.uint16)
    assert np.array_equal(got, want)
    assert (O.bf16_round(float("nan")) & 0x7fc0) == 0x7fc0
