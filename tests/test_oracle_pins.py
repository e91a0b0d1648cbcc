"""Pins of the reference oracle against what the paper and mathematics fix.

Each test checks the oracle against something other than itself: hand-worked
values of the paper's definitions (tests/golden), closed forms, invariants,
exact library reductions, brute force on tiny inputs, and the counts printed
in Table 1.  No GPU is needed.
"""
import itertools
import math
import os

import numpy as np
import pytest

from oracle import oracle as O
from oracle.sim import OracleRun
from tests.conftest import GOLDEN

EPS = 1e-8


def bf16_bits(values):
    """bf16 bit patterns of values that are exact in bf16 (checked)."""
    f = np.asarray(values, dtype=np.float32)
    bits = (f.view(np.uint32) >> 16).astype(np.uint16)
    back = (bits.astype(np.uint32) << 16).view(np.float32)
    assert np.array_equal(back, f, equal_nan=True), "value not exact in bf16"
    return bits


def rand_bf16(rng, n, scale=0.02):
    f = (rng.standard_normal(n) * scale).astype(np.float32)
    return (f.view(np.uint32) >> 16).astype(np.uint16)   # truncation: any bf16 pattern will do


# ----------------------------------------------------------------------------
# bf16 decoding
# ----------------------------------------------------------------------------

def test_bf16_value_known_patterns(oracle_lib):
    # bf16 = sign | 8-bit exponent (bias 127) | 7-bit mantissa.
    assert O.bf16_value(0x3F80) == 1.0
    assert O.bf16_value(0xBF80) == -1.0
    assert O.bf16_value(0x4000) == 2.0
    assert O.bf16_value(0x3F00) == 0.5
    assert O.bf16_value(0x3FC0) == 1.5
    assert O.bf16_value(0x0001) == 2.0 ** -133          # smallest subnormal
    assert O.bf16_value(0x0080) == 2.0 ** -126          # smallest normal
    assert O.bf16_value(0x7F7F) == (2 - 2 ** -7) * 2.0 ** 127
    assert O.bf16_value(0x7F80) == math.inf
    assert O.bf16_value(0xFF80) == -math.inf
    assert math.isnan(O.bf16_value(0x7FC0))
    z = O.bf16_value(0x8000)
    assert z == 0.0 and math.copysign(1.0, z) < 0


def test_bf16_value_all_patterns_match_numpy_view(oracle_lib):
    bits = np.arange(0, 1 << 16, 4099, dtype=np.uint32)
    ref = (bits << 16).view(np.float32).astype(np.float64)
    got = np.array([O.bf16_value(int(b)) for b in bits])
    assert np.array_equal(got, ref, equal_nan=True)


# ----------------------------------------------------------------------------
# Eq. 1: hand cases
# ----------------------------------------------------------------------------

def _load_measure_cases():
    cases, expects = {}, []
    with open(os.path.join(GOLDEN, "measure_hand_cases.txt")) as fh:
        for line in fh:
            line = line.split("#", 1)[0].strip()
            if not line:
                continue
            tok = line.split()
            if tok[0] == "expect":
                expects.append((tok[1], int(tok[2]), float(tok[3]), float(tok[4]),
                                float(tok[5]), tok[6]))
            else:
                case, layer, tensor, kind = tok[0], int(tok[1]), int(tok[2]), tok[3]
                vals = [float(x) for x in tok[4:]]
                cases.setdefault(case, {}).setdefault(layer, {}).setdefault(tensor, {})[kind] = vals
    return cases, expects


def test_measure_hand_cases(oracle_lib):
    cases, expects = _load_measure_cases()
    assert len(expects) == 4
    for case, layer, d_exp, a_exp, n_exp, u_expr in expects:
        tensors = []
        for k in sorted(cases[case][layer]):
            tk = cases[case][layer][k]
            tensors.append(O.Tensor(bf16_bits(tk["W"]), bf16_bits(tk["R"])))
        d, a, n = O.layer_sums(tensors)
        assert (d, a, n) == (d_exp, a_exp, n_exp), case
        u_exp = eval(u_expr, {"__builtins__": {}}, {"EPS": EPS})
        assert O.update_measure(d, a, n, EPS) == u_exp, case


def test_threshold_tie_and_epsilon_h1(oracle_lib):
    # H1 layer B: u = 0.25/(1+eps).  tau = 0.25 is just above u (eps breaks
    # the tie), tau = u itself persists because Eq. 3 uses ">=".
    u = O.update_measure(0.5, 2.0, 2.0, EPS)
    assert u < 0.25
    for tau, want in ((0.25, 0), (0.25 / (1.0 + EPS), 1)):
        delta = np.zeros(1)
        tl = np.zeros(1, dtype=np.int64)
        mask, nsel, _ = O.select_step([u], delta, tl, tau, 1000, 1, O.SNAPSHOT)
        assert mask[0] == want and nsel == want


def test_unchanged_layer_measures_zero(oracle_lib):
    rng = np.random.default_rng(1)
    w = rand_bf16(rng, 1001)
    wf = rng.standard_normal(77).astype(np.float32)
    d, a, n = O.layer_sums([O.Tensor(w, w.copy()), O.Tensor(wf, wf.copy())])
    assert d == 0.0 and a > 0 and n == 1078
    assert O.update_measure(d, a, n, EPS) == 0.0


def test_zero_reference_layer_is_selected(oracle_lib):
    # H2 generalised: with R = 0 the denominator is eps_w alone.
    w = bf16_bits([0.0, 2.0 ** -10, -2.0 ** -10, 0.0])
    d, a, n = O.layer_sums([O.Tensor(w, np.zeros(4, np.uint16))])
    assert (d, a, n) == (2.0 ** -9, 0.0, 4.0)
    u = O.update_measure(d, a, n, EPS)
    assert u == (2.0 ** -9 / 4) / EPS
    mask, _, _ = O.select_step([u], np.zeros(1), np.zeros(1, np.int64), 1e-3, 100, 1)
    assert mask[0] == 1


# ----------------------------------------------------------------------------
# Eq. 1: exact reductions, invariants
# ----------------------------------------------------------------------------

@pytest.mark.parametrize("dtype", ["bf16", "f32"])
def test_sums_match_exactly_rounded_fsum(oracle_lib, dtype):
    rng = np.random.default_rng(7)
    n = 50_003
    if dtype == "bf16":
        w, r = rand_bf16(rng, n), rand_bf16(rng, n)
        wf = (w.astype(np.uint32) << 16).view(np.float32).astype(np.float64)
        rf = (r.astype(np.uint32) << 16).view(np.float32).astype(np.float64)
    else:
        w = (rng.standard_normal(n) * 0.02).astype(np.float32)
        r = (rng.standard_normal(n) * 0.02).astype(np.float32)
        wf, rf = w.astype(np.float64), r.astype(np.float64)
    d, a, cnt = O.layer_sums([O.Tensor(w, r)])
    # |w - r| is exact in binary64 for both input types; fsum rounds once.
    d_ref = math.fsum(abs(x - y) for x, y in zip(wf.tolist(), rf.tolist()))
    a_ref = math.fsum(abs(y) for y in rf.tolist())
    assert cnt == n
    assert abs(d - d_ref) <= 1e-12 * d_ref
    assert abs(a - a_ref) <= 1e-12 * a_ref


def test_power_of_two_scaling_is_invariant(oracle_lib):
    # With eps_w = 0, Eq. 1 is a ratio of means: scaling W and R by 2^k
    # scales both sums exactly, so u is unchanged bit for bit.
    rng = np.random.default_rng(3)
    w = (rng.standard_normal(999) * 0.02).astype(np.float32)
    r = (w + rng.standard_normal(999).astype(np.float32) * 1e-4).astype(np.float32)
    u0 = O.update_measure(*O.layer_sums([O.Tensor(w, r)]), 0.0)
    for k in (-20, -3, 5, 30):
        s = np.float32(2.0 ** k)
        u1 = O.update_measure(*O.layer_sums([O.Tensor(w * s, r * s)]), 0.0)
        assert u1 == u0


def test_sums_depend_on_reference_not_current_for_denominator(oracle_lib):
    # The denominator is mean |W(t-1)|: swapping W and R changes A but not D.
    w = bf16_bits([1.0, 3.0])
    r = bf16_bits([2.0, 4.0])
    d1, a1, _ = O.layer_sums([O.Tensor(w, r)])
    d2, a2, _ = O.layer_sums([O.Tensor(r, w)])
    assert d1 == d2 == 2.0 and a1 == 6.0 and a2 == 4.0
    r = bf16_bits([2.0, 2.0])
    w2 = bf16_bits([-1.0, -3.0])
    d3, a3, _ = O.layer_sums([O.Tensor(w2, r)])
    assert d3 == 8.0 and a3 == 4.0        # |(-1)-2| + |(-3)-2|, not |w|-|r|


def test_special_values_propagate(oracle_lib):
    w = bf16_bits([1.0, np.inf])
    r = bf16_bits([1.0, 1.0])
    d, a, n = O.layer_sums([O.Tensor(w, r)])
    assert d == math.inf
    assert not math.isfinite(O.update_measure(d, a, n, EPS))
    w = np.array([0x3F80, 0x7FC0], dtype=np.uint16)      # 1, nan
    d, a, n = O.layer_sums([O.Tensor(w, r)])
    assert math.isnan(d)


# ----------------------------------------------------------------------------
# Eq. 2-4 and the staleness guard
# ----------------------------------------------------------------------------

def _load_sequences():
    out = []
    with open(os.path.join(GOLDEN, "select_sequences.txt")) as fh:
        for line in fh:
            line = line.split("#", 1)[0].strip()
            if not line:
                continue
            head, us, masks = [p.split() for p in line.split("|")]
            out.append((head[0], head[1], float(head[2]), int(head[3]),
                        [float(x) for x in us], [int(x) for x in masks]))
    return out


def test_select_golden_sequences(oracle_lib):
    seqs = _load_sequences()
    assert len(seqs) == 8
    for name, mode, tau, kmax, us, want in seqs:
        delta = np.zeros(1)
        tl = np.zeros(1, dtype=np.int64)
        got = []
        for t, u in enumerate(us, start=1):
            m, _, _ = O.select_step([u], delta, tl, tau, kmax, t,
                                    O.ACCUMULATE if mode == "accumulate" else O.SNAPSHOT)
            got.append(int(m[0]))
            if m[0]:
                assert delta[0] == 0.0 and tl[0] == t, name
        assert got == want, name


def _history_decisions(us, tau, kmax, mode):
    """The selection rule restated over the whole history instead of the
    running accumulator: a step persists when the drift since the last
    persistence (sum of u in accumulate mode, the current u in snapshot
    mode) reaches tau, is not finite, or the staleness reached kmax."""
    last, out = 0, []
    for t in range(1, len(us) + 1):
        drift = math.fsum(us[last:t]) if mode == O.ACCUMULATE else us[t - 1]
        sel = (not math.isfinite(drift)) or drift >= tau or (t - last) >= kmax
        out.append(int(sel))
        if sel:
            last = t
    return out


def test_select_brute_force_against_history_rule(oracle_lib):
    tau = 0.5
    values = [0.0, tau / 2, tau, 2 * tau]    # exact binary fractions: sums are exact
    checked = 0
    for mode in (O.SNAPSHOT, O.ACCUMULATE):
        for kmax in range(0, 5):
            # one layer, six steps: every sequence
            for seq in itertools.product(values, repeat=6):
                delta = np.zeros(1)
                tl = np.zeros(1, dtype=np.int64)
                got = []
                for t, u in enumerate(seq, start=1):
                    m, _, _ = O.select_step([u], delta, tl, tau, kmax, t, mode)
                    got.append(int(m[0]))
                    if kmax >= 1:
                        assert t - tl[0] <= kmax - 1     # staleness bound after the step
                assert got == _history_decisions(list(seq), tau, kmax, mode)
                checked += 1
            # two layers, three steps: layers do not interact
            for seq in itertools.product(values, repeat=6):
                u2 = np.array(seq).reshape(3, 2)
                delta = np.zeros(2)
                tl = np.zeros(2, dtype=np.int64)
                got = []
                for t in range(1, 4):
                    m, nsel, _ = O.select_step(u2[t - 1], delta, tl, tau, kmax, t, mode)
                    assert nsel == int(m.sum())
                    got.append(m.copy())
                got = np.array(got)
                for l in range(2):
                    assert list(got[:, l]) == _history_decisions(list(u2[:, l]), tau, kmax, mode)
    assert checked == 2 * 5 * 4 ** 6


def test_tau_multiplier_embedding_threshold(oracle_lib):
    # §3.4.3: embeddings use a 10x larger base threshold.
    u = [5e-3, 5e-3]
    mask, _, _ = O.select_step(u, np.zeros(2), np.zeros(2, np.int64), 1e-3, 100, 1,
                               O.SNAPSHOT, tau_mult=[10.0, 1.0])
    assert list(mask) == [0, 1]


def test_table1_default_layer_writes(oracle_lib):
    # Persisting every layer at every event (S_max = 0) for 1692 events
    # writes 1692 x N layers -- the "Default" rows of Table 1.
    rows = []
    with open(os.path.join(GOLDEN, "table1_default_writes.txt")) as fh:
        for line in fh:
            line = line.split("#", 1)[0].strip()
            if line:
                name, n, dirs, writes = line.split()
                rows.append((name, int(n), int(dirs), int(writes)))
    assert len(rows) == 3
    for name, n, dirs, writes in rows:
        delta = np.zeros(n)
        tl = np.zeros(n, dtype=np.int64)
        total = 0
        for t in range(1, dirs + 1):
            _, nsel, _ = O.select_step(np.zeros(n), delta, tl, 1e-3, 0, t)
            total += nsel
        assert total == writes, name


def test_staleness_closed_form(oracle_lib):
    # §3.3: larger layers count proportionally more in the weighted average
    mx, wt = O.staleness([0, 5, 10], [3, 1, 2], 10)
    assert mx == 10 and wt == (3 * 10 + 1 * 5 + 2 * 0) / 6
    mx, wt = O.staleness([7, 7], [1000, 1], 9)
    assert mx == 2 and wt == 2.0
    mx, wt = O.staleness([4, 0], [1, 1000], 4)
    assert mx == 4 and wt == 4000 / 1001


def test_select_rejects_bad_arguments(oracle_lib):
    with pytest.raises(ValueError):
        O.select_step([0.0], np.zeros(1), np.zeros(1, np.int64), math.nan, 1, 1)
    with pytest.raises(ValueError):
        O.select_step([0.0], np.zeros(1), np.zeros(1, np.int64), 1.0, -1, 1)


# ----------------------------------------------------------------------------
# Full layer state: packing (§3.1) -- checked with an independent parser
# ----------------------------------------------------------------------------

def _random_layer(rng, spec):
    ts = []
    for n, dt, moments in spec:
        w = rand_bf16(rng, n) if dt == "bf16" else rng.standard_normal(n).astype(np.float32)
        m = rng.standard_normal(n).astype(np.float32) if moments else None
        v = np.abs(rng.standard_normal(n)).astype(np.float32) if moments else None
        ts.append(O.Tensor(w, None, m, v))
    return ts


SPEC = [(1, "bf16", True), (7, "bf16", True), (129, "f32", True), (300, "bf16", False),
        (64, "bf16", True)]


@pytest.mark.parametrize("align", [16, 256, 4096])
def test_pack_layout_by_independent_parse(oracle_lib, align):
    rng = np.random.default_rng(11)
    ts = _random_layer(rng, SPEC)
    block = O.pack_layer(ts, align)
    up = lambda x: -(-x // align) * align
    # walk the documented layout: all W, then all m, then all v
    off = 0
    for part in ("w", "m", "v"):
        for t in ts:
            a = getattr(t, part)
            nb = 0 if a is None else a.nbytes
            if nb:
                assert np.array_equal(block[off:off + nb], a.view(np.uint8)), part
            assert not block[off + nb:off + up(nb)].any(), "padding must be zero"
            assert off % align == 0
            off += up(nb)
    assert off == block.size == O.layer_block_bytes(ts, align)


def test_unpack_inverts_pack_and_checks_padding(oracle_lib):
    rng = np.random.default_rng(12)
    ts = _random_layer(rng, SPEC)
    block = O.pack_layer(ts, 256)
    outs = [O.Tensor(np.zeros_like(t.w), None,
                     None if t.m is None else np.zeros_like(t.m),
                     None if t.v is None else np.zeros_like(t.v)) for t in ts]
    O.unpack_layer(block, outs, 256)
    for t, o in zip(ts, outs):
        assert np.array_equal(t.w, o.w)
        if t.m is not None:
            assert np.array_equal(t.m, o.m) and np.array_equal(t.v, o.v)
    bad = block.copy()
    bad[2] = 1       # inside the padding of the first (2-byte) W section
    with pytest.raises(ValueError):
        O.unpack_layer(bad, outs, 256)
    with pytest.raises(ValueError):
        O.unpack_layer(block[:-256], outs, 256)


# ----------------------------------------------------------------------------
# Composite recovery (§3.5, Eq. 8)
# ----------------------------------------------------------------------------

def test_composite_pick_equals_replay(oracle_lib):
    rng = np.random.default_rng(5)
    for _ in range(200):
        nl = int(rng.integers(1, 5))
        nv = int(rng.integers(0, 12))
        layer = rng.integers(0, nl, nv)
        step = rng.integers(0, 8, nv)
        dur = rng.integers(0, 2, nv)
        for t_fail in range(-1, 9):
            pick = O.composite_pick(layer, step, dur, nl, t_fail)
            # replay: apply durable writes in (step, record) order up to t_fail
            state = [-1] * nl
            for i in sorted(range(nv), key=lambda i: (step[i], i)):
                if dur[i] and step[i] <= t_fail:
                    state[layer[i]] = i
            assert list(pick) == state


def _small_layout():
    # 3 layers: layer 0 two bf16 tensors, layer 1 one fp32, layer 2 one bf16 without moments
    tensor_layer = [0, 0, 1, 2]
    numels = [33, 8, 17, 5]
    dtypes = ["bf16", "bf16", "f32", "bf16"]
    moments = [True, True, True, False]
    return tensor_layer, numels, dtypes, moments


def _gen(rng, numels, dtypes, moments):
    W = [rand_bf16(rng, n) if d == "bf16" else rng.standard_normal(n).astype(np.float32) * 0.02
         for n, d in zip(numels, dtypes)]
    M = [rng.standard_normal(n).astype(np.float32) if mo else None for n, mo in zip(numels, moments)]
    V = [np.abs(rng.standard_normal(n)).astype(np.float32) if mo else None
         for n, mo in zip(numels, moments)]
    return W, M, V


def test_composite_equals_latest_persisted_versions(oracle_lib):
    tl, numels, dtypes, moments = _small_layout()
    rng = np.random.default_rng(9)
    run = OracleRun(tl, numels, 3, dtypes, moments)
    W, M, V = _gen(rng, numels, dtypes, moments)
    run.set_reference(W)
    history = {}          # (layer, step) -> copies of that layer's tensors
    mask0, _, _ = O.select_step(np.zeros(3), run.delta, run.t_last, 1.0, 0, 0)
    assert mask0.all()
    for t in range(0, 9):
        if t > 0:
            W, M, V = _gen(rng, numels, dtypes, moments)
            u, _ = run.measure(W)
            mask = run.select(u, 1e-3, 3, t)
        else:
            mask = mask0
        run.pack(mask, W, M, V, t)
        run.commit(mask, W)
        run.mark_durable(t)
        for l in range(3):
            if mask[l]:
                history[(l, t)] = [(W[k].copy(), None if M[k] is None else M[k].copy(),
                                    None if V[k] is None else V[k].copy())
                                   for k in run.layer_tensors[l]]
    for t_fail in range(0, 9):
        comp, pick = run.composite(t_fail)
        for l in range(3):
            t_l = max(s for (ll, s) in history if ll == l and s <= t_fail)
            assert run.versions[pick[l]]["step"] == t_l
            for k, (w, m, v) in zip(run.layer_tensors[l], history[(l, t_l)]):
                assert np.array_equal(comp[k][0], w)
                assert (m is None) or (np.array_equal(comp[k][1], m) and np.array_equal(comp[k][2], v))
    # snapshot mode: the reference is exactly the newest composite's weights
    comp, _ = run.composite(8)
    for k in range(len(numels)):
        assert np.array_equal(comp[k][0], run.R[k])


def test_crash_before_durable_uses_previous_version(oracle_lib):
    tl, numels, dtypes, moments = _small_layout()
    rng = np.random.default_rng(10)
    run = OracleRun(tl, numels, 3, dtypes, moments)
    W0, M0, V0 = _gen(rng, numels, dtypes, moments)
    run.set_reference(W0)
    allmask = np.ones(3, np.uint8)
    run.pack(allmask, W0, M0, V0, 0)
    run.mark_durable(0)
    W1, M1, V1 = _gen(rng, numels, dtypes, moments)
    run.pack(allmask, W1, M1, V1, 1)      # never becomes durable
    run.drop_pending()
    comp, pick = run.composite(1)
    assert all(run.versions[p]["step"] == 0 for p in pick)
    for k in range(len(numels)):
        assert np.array_equal(comp[k][0], W0[k])


def test_staleness_bound_holds_over_random_runs(oracle_lib):
    # §3.3 invariant: with S_max = K no layer is ever more than K steps stale
    # at a failure point, whatever the drift.
    rng = np.random.default_rng(4)
    for K in (1, 2, 5):
        delta = np.zeros(6)
        tl = np.zeros(6, dtype=np.int64)
        for t in range(1, 60):
            u = rng.choice([0.0, 1e-4, 1e-3, 5e-3], size=6)
            O.select_step(u, delta, tl, 1e-3, K, t, O.ACCUMULATE)
            assert (t - tl).max() <= K - 1
            assert (t + 1 - tl).max() <= K    # a failure before the next opportunity
