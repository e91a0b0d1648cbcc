"""Host-side checks of the synthetic workloads: the layer partition of §2.2
against the layer counts printed in Table 1, exact parameter counts of the
five workloads, and reproducible seeding."""
import numpy as np
import pytest

from lc_workloads import gen, shapes
from lc_workloads.configs import WORKLOADS


def test_layer_partition_matches_table1_counts():
    # Table 1 lists Qwen2.5-7B with 31 layers, Qwen2.5-3B with 38 and
    # Llama3.2-1B with 18; N = B + 3 with an untied head, B + 2 when tied.
    qwen7b = shapes.decoder_shape("qwen2.5-7b", 28, 3584, 18944, 28, 4, 128, 152064, tied=False)
    qwen3b = shapes.decoder_shape("qwen2.5-3b", 36, 2048, 11008, 16, 2, 128, 151936, tied=True)
    assert qwen7b.nlayers == 31
    assert qwen3b.nlayers == 38
    assert shapes.llama32_1b().nlayers == 18
    assert qwen7b.layer_names[0] == "embed_tokens" and qwen7b.layer_names[-1] == "lm_head"
    assert qwen7b.layer_names[-2] == "norm"


def test_parameter_counts():
    assert shapes.tiny().numel == 6_244_608
    assert shapes.llama32_1b().numel == 1_235_814_400
    b8 = shapes.llama3_8b()
    assert b8.numel == 8_030_261_248 and b8.nlayers == 35 and len(b8.tensors) == 291
    per = shapes.llama3_8b(per_tensor=True)
    assert per.nlayers == 291 and per.numel == b8.numel
    sizes = sorted(t.numel for t in per.tensors)
    assert sizes[0] == 4096 and sizes[-1] == 525_336_576


def test_seeding_is_reproducible_and_distinct():
    torch = pytest.importorskip("torch")
    a = gen.SyntheticState(shapes.tiny(), device="cpu", seed=3)
    b = gen.SyntheticState(shapes.tiny(), device="cpu", seed=3)
    c = gen.SyntheticState(shapes.tiny(), device="cpu", seed=4)
    for k in (0, 5, 37):
        assert torch.equal(a.W[k], b.W[k]) and torch.equal(a.m[k], b.m[k])
        assert not torch.equal(a.W[k], c.W[k])
        assert torch.equal(a.W[k], a.R[k])
    a.drift(1, np.full(6, 1e-2))
    b.drift(1, np.full(6, 1e-2))
    assert all(torch.equal(x, y) for x, y in zip(a.W, b.W))
    assert any(not torch.equal(x, y) for x, y in zip(a.W, a.R))
    assert len({gen.mix_seed(0, s, k, 1) for s in range(20) for k in range(20)}) == 400


def test_flat_and_skew_allocations_misalign():
    pytest.importorskip("torch")
    spec = shapes.tiny()
    f = gen.SyntheticState(spec, device="cpu", seed=0, alloc="flat")
    s = gen.SyntheticState(spec, device="cpu", seed=0, alloc="skew")
    assert all(w.data_ptr() % 16 == r.data_ptr() % 16 for w, r in zip(f.W, f.R))
    assert any(w.data_ptr() % 16 != r.data_ptr() % 16 for w, r in zip(s.W, s.R))


def test_calibration_targets_quarter_of_layers():
    for name in ("1b", "8b"):
        wl = WORKLOADS[name]
        sc = wl.layer_scales(wl.shape())
        f = gen.expected_fraction(sc, wl.tau, wl.max_staleness)
        assert abs(f - 0.25) < 0.02, (name, f)


def test_flat_views_never_overlap():
    pytest.importorskip("torch")
    spec = shapes.tiny()
    for alloc in ("flat", "skew"):
        st = gen.SyntheticState(spec, device="cpu", seed=0, alloc=alloc)
        for kind in ("W", "R", "m", "v"):
            spans = sorted((t.data_ptr(), t.data_ptr() + t.numel() * t.element_size())
                           for t in getattr(st, kind) if t is not None)
            assert all(a[1] <= b[0] for a, b in zip(spans, spans[1:])), (alloc, kind)
