"""GPU parity of the fused AdamW + drift step (§3.4.2: the drift of Eq. 1
is read off the optimizer update; Eq. 2 accumulates it) against the oracle,
through the C ABI: updated weights, moments and bf16 model copy bit for bit,
u within 1e-5, selections and packed full layer states exact."""
import numpy as np
import pytest

from lc_workloads.gen import mix_seed
from oracle import oracle as O
from tests.lc_harness import U_RTOL, rel_err, require_gpu

pytestmark = pytest.mark.gpu

HP = (2e-3, 0.9, 0.999, 1e-8, 0.01)     # lr, beta1, beta2, eps, weight decay


class FusedState:
    """fp32 master weights, moments, gradients and bf16 model copies.

    layout "separate": one allocation per tensor; "flat": back to back in
    shared buffers (misaligned starts); "skew": the gradients additionally
    shifted by one element, so they never line up with the weights."""

    def __init__(self, sizes_layers, layout, grad_dtype, seed=0):
        import torch
        self.torch = torch
        self.specs = list(sizes_layers)
        self.nlayers = max(l for _, l in self.specs) + 1
        n = [s for s, _ in self.specs]
        total = sum(n) + 64
        gdt = torch.bfloat16 if grad_dtype == "bf16" else torch.float32
        if layout == "separate":
            mk = lambda dt: [torch.empty(k, dtype=dt, device="cuda") for k in n]
            self.p, self.m, self.v = mk(torch.float32), mk(torch.float32), mk(torch.float32)
            self.g, self.model = mk(gdt), mk(torch.bfloat16)
        else:
            bufs = {name: torch.empty(total, dtype=dt, device="cuda")
                    for name, dt in (("p", torch.float32), ("m", torch.float32), ("v", torch.float32),
                                     ("g", gdt), ("model", torch.bfloat16))}
            shift = {"g": 1 if layout == "skew" else 0}
            views = {k: [] for k in bufs}
            off = 0
            for k in n:
                for name, b in bufs.items():
                    s = off + shift.get(name, 0)
                    views[name].append(b[s:s + k])
                off += k
            self.p, self.m, self.v, self.g, self.model = (views[x] for x in ("p", "m", "v", "g", "model"))
            self._bufs = bufs
        gen = torch.Generator(device="cuda")
        for i, k in enumerate(n):
            gen.manual_seed(mix_seed(seed, 0, i, 0))
            self.p[i].normal_(0.0, 0.02, generator=gen)
            self.m[i].normal_(0.0, 1e-3, generator=gen)
            self.v[i].normal_(0.0, 1e-6, generator=gen).abs_()
        self.seed = seed

    def new_grads(self, step):
        gen = self.torch.Generator(device="cuda")
        for i, g in enumerate(self.g):
            gen.manual_seed(mix_seed(self.seed, step, i, 1))
            scale = 1e-3 * (1 + self.specs[i][1])
            g.copy_(self.torch.randn(g.numel(), generator=gen, device="cuda") * scale)

    @staticmethod
    def host(t):
        import torch
        if t.dtype == torch.bfloat16:
            return t.view(torch.int16).cpu().numpy().view(np.uint16).copy()
        return t.cpu().numpy().copy()


def _run(sizes_layers, layout, grad_dtype, steps=4, tau=0.2, K=3, engine="bulk"):
    torch = require_gpu()
    import paper_2609_27193_gb300 as P
    st = FusedState(sizes_layers, layout, grad_dtype)
    lc = P.LayerCheck(mode=P.LC_DRIFT_ACCUMULATE, copy_engine=engine)
    lc.register_layout([P.segment(l, st.p[i], None, st.m[i], st.v[i])
                        for i, (_, l) in enumerate(st.specs)], st.nlayers)
    lc.register_optimizer(st.g, st.model)
    delta = np.zeros(st.nlayers)
    t_last = np.zeros(st.nlayers, dtype=np.int64)
    for t in range(1, steps + 1):
        st.new_grads(t)
        torch.cuda.synchronize()
        # oracle inputs: the state before the step
        P0 = [st.host(x) for x in st.p]
        M0 = [st.host(x) for x in st.m]
        V0 = [st.host(x) for x in st.v]
        G = [st.host(x) for x in st.g]
        lc.adamw_step_measure(t, *HP[:1], beta1=HP[1], beta2=HP[2], eps=HP[3], weight_decay=HP[4])
        mask, u, nbytes = lc.select(tau, K)
        torch.cuda.synchronize()
        sums = np.zeros((st.nlayers, 3))
        models = []
        for i, (n, l) in enumerate(st.specs):
            model = np.zeros(n, np.uint16)
            d, a = O.adamw_step(HP, t, P0[i], M0[i], V0[i], G[i], model)
            models.append(model)
            sums[l] += (d, a, n)
            assert np.array_equal(st.host(st.p[i]), P0[i]), "weights of tensor %d, step %d" % (i, t)
            assert np.array_equal(st.host(st.m[i]), M0[i]), "exp_avg of tensor %d" % i
            assert np.array_equal(st.host(st.v[i]), V0[i]), "exp_avg_sq of tensor %d" % i
            assert np.array_equal(st.host(st.model[i]), model), "model copy of tensor %d" % i
        ou = np.array([O.update_measure(d, a, n, 1e-8) for d, a, n in sums])
        assert rel_err(u, ou).max() <= U_RTOL, rel_err(u, ou)
        acc = delta + ou
        omask, _, _ = O.select_step(ou, delta, t_last, tau, K, t, O.ACCUMULATE)
        band = np.abs(acc - tau) <= U_RTOL * tau
        bad = np.flatnonzero((mask != omask) & ~band)
        assert bad.size == 0, "selection differs on layers %s at step %d" % (bad, t)
        for l in np.flatnonzero(mask != omask):      # adopt the device decision in the band
            if mask[l]:
                delta[l], t_last[l] = 0.0, t
            else:
                delta[l], t_last[l] = acc[l], t_last[l]
        # the full layer state of the persisted layers, fp32 master weights
        dst = torch.empty(max(16, nbytes), dtype=torch.uint8, device="cuda")
        lc.pack_device(dst)
        lc.commit_snapshot()
        torch.cuda.synchronize()
        got = dst.cpu().numpy()
        off = lc.offsets()
        for l in np.flatnonzero(mask):
            ts = [O.Tensor(P0[i], None, M0[i], V0[i]) for i, (_, ll) in enumerate(st.specs) if ll == l]
            block = O.pack_layer(ts)
            assert np.array_equal(got[int(off[l]):int(off[l]) + block.size], block), "block %d" % l
    assert lc.counters()["bulk_measure_launches"] == (steps if engine == "bulk" else 0)
    lc.close()
    return mask


SIZES = [(1, 0), (7, 0), (4095, 1), (4099, 1), (100003, 2), (65536, 3), (3, 3), (250001, 4)]


@pytest.mark.parametrize("engine", ["bulk", "threads"])
@pytest.mark.parametrize("layout", ["separate", "flat", "skew"])
@pytest.mark.parametrize("grad_dtype", ["bf16", "f32"])
def test_fused_adamw_bit_exact(layout, grad_dtype, engine):
    """Both engines: the bulk-load step takes chunks of 512 vectors of the
    separate allocations (the 250,001- and 100,003-parameter segments span
    several chunks and end in a partial vector); "flat" starts tensors on
    odd offsets, so bf16 gradient vectors begin off 16 bytes and are peeled;
    "skew" never lines up and goes element by element."""
    _run(SIZES, layout, grad_dtype, engine=engine)


def test_fused_step_requires_accumulate_mode_and_fp32_weights():
    torch = require_gpu()
    import paper_2609_27193_gb300 as P
    st = FusedState([(64, 0)], "separate", "bf16")
    lc = P.LayerCheck()                      # snapshot mode
    r = torch.empty(64, dtype=torch.float32, device="cuda")
    lc.register_layout([P.segment(0, st.p[0], r, st.m[0], st.v[0])], 1)
    with pytest.raises(P.LCError) as e:
        lc.register_optimizer(st.g)
    assert e.value.status == 2
    lc.close()
    lc = P.LayerCheck(mode=P.LC_DRIFT_ACCUMULATE)
    lc.register_layout([P.segment(0, st.p[0], None, st.m[0], st.v[0])], 1)
    with pytest.raises(P.LCError) as e:
        lc.measure(1)                        # no snapshot to measure against
    assert e.value.status == 2
    with pytest.raises(P.LCError) as e:
        lc.adamw_step_measure(1, 1e-3)       # no optimizer registered yet
    assert e.value.status == 2
    lc.register_optimizer(st.g, st.model)
    with pytest.raises(P.LCError):
        lc.adamw_step_measure(0, 1e-3)       # bias correction needs t >= 1
    with pytest.raises(P.LCError):
        lc.adamw_step_measure(1, 1e-3, beta1=1.0)
    lc.adamw_step_measure(1, 1e-3)
    lc.select(1e-3, 8)
    lc.close()


def test_bulk_fused_step_wait_bound_reports_timeout():
    """LC_DEBUG_MEASURE_STALL on the bulk-load fused step: each CTA's first
    chunk announces 16 bytes that never arrive, the bounded waits run out,
    and lc_select fails with LC_ERR_TIMEOUT; a fresh context still steps."""
    import time
    torch = require_gpu()
    import paper_2609_27193_gb300 as P
    st = FusedState([(250001, 0), (65536, 1)], "separate", "bf16")
    lc = P.LayerCheck(mode=P.LC_DRIFT_ACCUMULATE, debug_flags=P.LC_DEBUG_MEASURE_STALL)
    lc.register_layout([P.segment(l, st.p[i], None, st.m[i], st.v[i]) for i, (_, l) in enumerate(st.specs)],
                       st.nlayers)
    lc.register_optimizer(st.g, st.model)
    st.new_grads(1)
    t0 = time.perf_counter()
    lc.adamw_step_measure(1, 1e-3)
    with pytest.raises(P.LCError) as e:
        lc.select(1e-3, 8)
    assert e.value.status == 6
    assert time.perf_counter() - t0 < 30.0
    assert lc.counters()["bulk_measure_launches"] == 1
    lc.close()
    torch.cuda.synchronize()
    _run([(4099, 0), (65536, 1)], "separate", "bf16", steps=2)
