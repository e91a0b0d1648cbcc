"""The five synthetic workloads (shapes, thresholds, drift recipes).

tiny        4 blocks d=256, tied head; s_l log-uniform in [1e-5, 1e-2];
            tau = 1e-3, S_max = 4, 20 steps, seed 0.
1b          Llama-3.2-1B shape; s_l log-uniform over one decade, scaled so
            that about 25% of the layers persist per step; tau = 1e-3,
            S_max = 8, 50 steps.
8b          Llama-3-8B shape (35 layers); log s_l a U-shape over depth plus
            N(0, 0.3) log-noise, scaled to about 25% persisted per step at
            tau = 1e-3; tau in {5e-4, 1e-3, 2e-3}, S_max = 8, 100 steps.
8b-tensor   the same 291 tensors, each its own unit; s log-uniform in
            [1e-6, 1e-2] per tensor; tau = 1e-3, S_max = 16.
8b-cadence  the 8b layout for 200 steps with drift regimes switching every
            50 steps (uniform, top-heavy, bottom-heavy, sparse 10%), beside a
            looping bf16 8192^3 matmul on another stream.
"""
from dataclasses import dataclass, field
from typing import Callable, List, Optional

import numpy as np

from . import gen, shapes


@dataclass
class Workload:
    name: str
    shape_fn: Callable
    tau: float
    max_staleness: int
    steps: int
    seed: int
    scales: Callable            # (shape, rng, tau, K) -> per-layer scales
    taus: List[float] = field(default_factory=list)
    regimes: Optional[List[str]] = None

    def shape(self):
        return self.shape_fn()

    def layer_scales(self, shape):
        rng = np.random.default_rng(self.seed + 1000)
        return np.asarray(self.scales(shape, rng, self.tau, self.max_staleness), dtype=np.float64)


def _tiny_scales(shape, rng, tau, K):
    return gen.loguniform(shape.nlayers, 1e-5, 1e-2, rng)


def _b1_scales(shape, rng, tau, K):
    base = gen.loguniform(shape.nlayers, 1.0, 10.0, rng)
    return base * gen.calibrate(base, tau, K, 0.25)


def _b8_scales(shape, rng, tau, K):
    base = gen.u_shape(shape.nlayers, 8.0, 1.0, 0.3, rng)
    return base * gen.calibrate(base, tau, K, 0.25)


def _tensor_scales(shape, rng, tau, K):
    return gen.loguniform(shape.nlayers, 1e-6, 1e-2, rng)


WORKLOADS = {
    "tiny": Workload("tiny", shapes.tiny, 1e-3, 4, 20, 0, _tiny_scales),
    "1b": Workload("1b", shapes.llama32_1b, 1e-3, 8, 50, 0, _b1_scales),
    "8b": Workload("8b", shapes.llama3_8b, 1e-3, 8, 100, 0, _b8_scales,
                   taus=[5e-4, 1e-3, 2e-3]),
    "8b-tensor": Workload("8b-tensor", lambda: shapes.llama3_8b(per_tensor=True), 1e-3, 16, 100, 0,
                          _tensor_scales),
    "8b-cadence": Workload("8b-cadence", shapes.llama3_8b, 1e-3, 8, 200, 0, _b8_scales,
                           regimes=["uniform", "top_heavy", "bottom_heavy", "sparse"]),
}


def cadence_scales(workload, shape, step):
    """Scales of the regime active at `step` (regimes switch every 50 steps)."""
    regime = workload.regimes[min(len(workload.regimes) - 1, (max(step, 1) - 1) // 50)]
    rng = np.random.default_rng(workload.seed + 2000 + (max(step, 1) - 1) // 50)
    return gen.regime_scales(regime, shape.nlayers, workload.tau, rng), regime
