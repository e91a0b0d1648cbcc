"""Seeded synthetic inputs for the LayerCheck path (no method arithmetic).

A workload is a set of parameter tensors with fp32 master weights M, the
model weights W = round(M) (bf16, round-to-nearest-even, or fp32 = M), the
reference snapshot R, and fp32 Adam moments m, v.  Initial state: M ~
N(0, 0.02), R = W, m ~ N(0, 1e-3), v = |N(0, 1e-6)|.  A training step adds
N(0, (s_l * 0.02)^2) noise to M for every tensor of layer l and, by default,
redraws m and v, so persisted versions of different steps differ.  Random
numbers come from torch generators seeded per (seed, step, tensor, stream)
with splitmix64, so a given device type reproduces them exactly.
"""
import math

import numpy as np
import torch

_MASK64 = (1 << 64) - 1


def mix_seed(*parts):
    """splitmix64 over the parts -> a 63-bit torch seed."""
    x = 0x9E3779B97F4A7C15
    for p in parts:
        x = (x + (int(p) & _MASK64) + 0x9E3779B97F4A7C15) & _MASK64
        z = x
        z = ((z ^ (z >> 30)) * 0xBF58476D1CE4E5B9) & _MASK64
        z = ((z ^ (z >> 27)) * 0x94D049BB133111EB) & _MASK64
        x = z ^ (z >> 31)
    return x & ((1 << 63) - 1)


def _gen(device, *parts):
    g = torch.Generator(device=device)
    g.manual_seed(mix_seed(*parts))
    return g


class SyntheticState:
    """Device tensors of one workload.

    master=False keeps no fp32 master copy (a smaller footprint for kernel
    captures): the drift is then rounded into W at every step.
    snapshot=False allocates no reference snapshot R (the fused optimizer
    path measures the update itself).
    alloc: "separate" -- one allocation per tensor (16-byte aligned);
           "flat"     -- one buffer per kind, tensors back to back, so a
                         tensor after an odd-sized one starts misaligned;
           "skew"     -- like "flat" but R's buffer is shifted by one element,
                         so W and R are never co-aligned.
    """

    def __init__(self, shape, device="cuda", seed=0, alloc="separate", moments=True,
                 dtypes=None, moments_mask=None, master=True, snapshot=True):
        self.shape = shape
        self.device = torch.device(device)
        self.seed = int(seed)
        self.alloc = alloc
        self.specs = list(shape.tensors)
        nt = len(self.specs)
        self.dtypes = list(dtypes) if dtypes is not None else [t.dtype for t in self.specs]
        self.has_moments = ([bool(moments)] * nt if moments_mask is None else
                            [bool(moments) and bool(x) for x in moments_mask])
        self.master = bool(master)
        self.snapshot = bool(snapshot)
        self.W, self.R, self.M, self.m, self.v = [], [], [], [], []
        self._allocate()
        self.init()

    @property
    def nlayers(self):
        return self.shape.nlayers

    @property
    def tensor_layer(self):
        return [t.layer for t in self.specs]

    @property
    def numels(self):
        return [t.numel for t in self.specs]

    def _tdtype(self, k):
        return torch.bfloat16 if self.dtypes[k] == "bf16" else torch.float32

    def _allocate(self):
        dev = self.device
        nt = len(self.specs)
        if self.alloc == "separate":
            for k, t in enumerate(self.specs):
                self.W.append(torch.empty(t.numel, dtype=self._tdtype(k), device=dev))
                self.R.append(torch.empty(t.numel, dtype=self._tdtype(k), device=dev)
                              if self.snapshot else None)
                self.M.append(torch.empty(t.numel, dtype=torch.float32, device=dev)
                              if self.master else None)
                mo = self.has_moments[k]
                self.m.append(torch.empty(t.numel, dtype=torch.float32, device=dev) if mo else None)
                self.v.append(torch.empty(t.numel, dtype=torch.float32, device=dev) if mo else None)
            return
        if self.alloc not in ("flat", "skew"):
            raise ValueError("unknown alloc %r" % self.alloc)
        # byte offsets of each tensor in the flat weight buffers; "skew" leaves
        # a 16-byte gap after every tensor so the shifted R views never overlap
        gap = 16 if self.alloc == "skew" else 0
        offs, o = [], 0
        for k, t in enumerate(self.specs):
            esz = 2 if self.dtypes[k] == "bf16" else 4
            o = -(-o // esz) * esz
            offs.append(o)
            o += t.numel * esz + gap
        total = o + 64
        shift = 2 if self.alloc == "skew" else 0
        wbuf = torch.empty(total, dtype=torch.uint8, device=dev)
        rbuf = torch.empty(total + 16, dtype=torch.uint8, device=dev)
        mtot = sum(t.numel for t in self.specs) + 16
        mbuf = torch.empty(mtot, dtype=torch.float32, device=dev)
        vbuf = torch.empty(mtot, dtype=torch.float32, device=dev)
        fo = 0
        for k, t in enumerate(self.specs):
            esz = 2 if self.dtypes[k] == "bf16" else 4
            # a shift of 2 bytes breaks 4-byte alignment of fp32 tensors; keep
            # them element-aligned by shifting those by 4
            sh = shift if esz == 2 else (4 if shift else 0)
            b0 = offs[k]
            self.W.append(wbuf[b0:b0 + t.numel * esz].view(self._tdtype(k)))
            self.R.append(rbuf[b0 + sh:b0 + sh + t.numel * esz].view(self._tdtype(k)))
            self.M.append(torch.empty(t.numel, dtype=torch.float32, device=dev)
                          if self.master else None)
            if self.has_moments[k]:
                self.m.append(mbuf[fo:fo + t.numel])
                self.v.append(vbuf[fo:fo + t.numel])
            else:
                self.m.append(None)
                self.v.append(None)
            fo += t.numel
        self._buffers = (wbuf, rbuf, mbuf, vbuf)

    def init(self):
        """Step-0 state: M ~ N(0, 0.02), W = round(M), R = W, fresh moments."""
        with torch.no_grad():
            for k in range(len(self.specs)):
                g = _gen(self.device, self.seed, 0, k, 0)
                if self.master:
                    self.M[k].normal_(0.0, 0.02, generator=g)
                    self.W[k].copy_(self.M[k])
                else:
                    self.W[k].normal_(0.0, 0.02, generator=g)
                if self.R[k] is not None:
                    self.R[k].copy_(self.W[k])
                self._draw_moments(0, k)

    def _draw_moments(self, step, k):
        if not self.has_moments[k]:
            return
        self.m[k].normal_(0.0, 1e-3, generator=_gen(self.device, self.seed, step, k, 2))
        self.v[k].normal_(0.0, 1e-6, generator=_gen(self.device, self.seed, step, k, 3)).abs_()

    def drift(self, step, layer_scale, redraw_moments=True, tensor_scale=None):
        """One synthetic training step: M += N(0, (s*0.02)^2), W = round(M)."""
        with torch.no_grad():
            for k, t in enumerate(self.specs):
                s = float(tensor_scale[k] if tensor_scale is not None else layer_scale[t.layer])
                if s > 0.0:
                    g = _gen(self.device, self.seed, step, k, 1)
                    noise = torch.randn(t.numel, generator=g, device=self.device, dtype=torch.float32)
                    if self.master:
                        self.M[k].add_(noise, alpha=s * 0.02)
                        self.W[k].copy_(self.M[k])
                    else:      # lean mode: the drift is rounded into W every step
                        self.W[k].add_(noise.mul_(s * 0.02).to(self.W[k].dtype))
                    del noise
                if redraw_moments:
                    self._draw_moments(step, k)

    def resync_master(self):
        """After a recovery wrote W on the device: the fp32 master copy
        restarts from the restored weights."""
        if not self.master:
            return
        with torch.no_grad():
            for k in range(len(self.specs)):
                self.M[k].copy_(self.W[k])

    def set_values(self, k, w=None, r=None):
        """Overwrite W (and M) and/or R of tensor k with given float values."""
        with torch.no_grad():
            if w is not None:
                if self.master:
                    self.M[k].copy_(torch.as_tensor(w, dtype=torch.float32))
                    self.W[k].copy_(self.M[k])
                else:
                    self.W[k].copy_(torch.as_tensor(w, dtype=torch.float32))
            if r is not None:
                self.R[k].copy_(torch.as_tensor(r, dtype=torch.float32))

    # -- host copies for the oracle (numpy; bf16 as uint16 bit patterns) --
    @staticmethod
    def to_numpy(t):
        if t is None:
            return None
        if t.dtype == torch.bfloat16:
            return t.detach().view(torch.int16).cpu().numpy().view(np.uint16)
        return t.detach().cpu().numpy()

    def host(self, kind, k):
        return self.to_numpy(getattr(self, kind)[k])

    def host_all(self, kind):
        return [self.host(kind, k) for k in range(len(self.specs))]

    def bytes_resident(self):
        tot = 0
        for lst in (self.W, self.R, self.M, self.m, self.v):
            for t in lst:
                if t is not None:
                    tot += t.numel() * t.element_size()
        return tot


# --------------------------------------------------------------------------
# drift scales s_l
# --------------------------------------------------------------------------

def loguniform(n, lo, hi, rng):
    return np.exp(rng.uniform(math.log(lo), math.log(hi), n))


def u_shape(n, s_edge, s_mid, noise_sigma, rng):
    """log s over depth is a parabola, largest at the first and last layers,
    plus N(0, noise_sigma) natural-log noise."""
    x = np.linspace(-1.0, 1.0, n)
    logs = math.log(s_mid) + (math.log(s_edge) - math.log(s_mid)) * x * x
    return np.exp(logs + rng.normal(0.0, noise_sigma, n))


def expected_fraction(scales, tau, max_staleness):
    """Fraction of layers persisted per step if a layer of scale s reaches
    drift s * sqrt(k) after k steps (a random walk in M, measured against
    the snapshot) and the staleness guard forces it after K steps."""
    s = np.asarray(scales, dtype=np.float64)
    with np.errstate(divide="ignore"):
        k = np.ceil((tau / np.maximum(s, 1e-300)) ** 2)
    period = np.clip(k, 1, max(1, max_staleness))
    return float(np.mean(1.0 / period))


def calibrate(scales, tau, max_staleness, target):
    """Common factor c such that expected_fraction(c * scales) ~= target."""
    lo, hi = 1e-6, 1e6
    for _ in range(200):
        mid = math.sqrt(lo * hi)
        if expected_fraction(scales * mid, tau, max_staleness) < target:
            lo = mid
        else:
            hi = mid
    return math.sqrt(lo * hi)


def regime_scales(regime, n, tau, rng):
    """Per-layer scales of the cadence workload's regimes."""
    if regime == "uniform":
        return np.full(n, tau / 2.0)
    x = np.linspace(0.0, 1.0, n)
    if regime == "top_heavy":
        return tau * np.exp(math.log(1 / 8) + math.log(16) * x)
    if regime == "bottom_heavy":
        return tau * np.exp(math.log(2) - math.log(16) * x)
    if regime == "sparse":
        s = np.full(n, tau / 50.0)
        hot = rng.choice(n, size=max(1, n // 10), replace=False)
        s[hot] = 2.0 * tau
        return s
    raise ValueError(regime)
