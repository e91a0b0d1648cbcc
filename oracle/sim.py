"""Multi-step oracle run (TEST INFRASTRUCTURE ONLY).

Drives the C restatements of lc_oracle.c through the per-step procedure of
§3.1-§3.5: at every checkpoint opportunity measure each layer (Eq. 1),
update the accumulators and select (Eq. 2-4, §3.3 staleness guard), persist
the full state of the selected layers (§3.1), commit their reference
snapshot, and on recovery assemble the mixed-timestamp composite (§3.5,
Eq. 8).  The oracle keeps its own reference copies, accumulators, last
persistence steps and version store; nothing here is read back from the
CUDA path.
"""
import hashlib

import numpy as np

from . import oracle as O


def digest(block):
    return hashlib.blake2b(memoryview(np.ascontiguousarray(block)), digest_size=16).hexdigest()


class OracleRun:
    """State of the method over a fixed layout.

    tensor_layer[k] is the layer id of tensor k (registration order);
    numels[k], dtypes[k] ('bf16' or 'f32') and has_moments[k] describe it.
    keep_blocks: "all" keeps every persisted block (any restore point),
    "latest" keeps only each layer's newest block (restore at the newest
    step only) plus a digest of every version.
    """

    def __init__(self, tensor_layer, numels, nlayers, dtypes=None, has_moments=None,
                 eps_w=1e-8, mode=O.SNAPSHOT, align=256, tau_mult=None, keep_blocks="all"):
        self.tensor_layer = [int(l) for l in tensor_layer]
        self.numels = [int(n) for n in numels]
        self.nlayers = int(nlayers)
        nt = len(self.tensor_layer)
        self.dtypes = list(dtypes) if dtypes is not None else ["bf16"] * nt
        self.has_moments = list(has_moments) if has_moments is not None else [True] * nt
        self.eps_w, self.mode, self.align = float(eps_w), int(mode), int(align)
        self.tau_mult = None if tau_mult is None else np.asarray(tau_mult, dtype=np.float64)
        self.keep_blocks = keep_blocks
        self.layer_tensors = [[k for k in range(nt) if self.tensor_layer[k] == l]
                              for l in range(self.nlayers)]
        self.layer_numel = np.array([sum(self.numels[k] for k in ks) for ks in self.layer_tensors],
                                    dtype=np.int64)
        self.R = [None] * nt
        self.delta = np.zeros(self.nlayers, dtype=np.float64)
        self.t_last = np.zeros(self.nlayers, dtype=np.int64)
        self.versions = []       # dicts: layer, step, durable, digest, nbytes
        self.blocks = {}         # version index -> block (kept per keep_blocks)
        self.last_acc = None

    # -- inputs ---------------------------------------------------------
    def set_reference(self, R):
        """Initial reference weights (the base state, §3.4.3 warm-up)."""
        self.R = [np.array(r, copy=True) for r in R]

    def _tensors(self, l, W, M=None, V=None):
        out = []
        for k in self.layer_tensors[l]:
            m = M[k] if (M is not None and self.has_moments[k]) else None
            v = V[k] if (V is not None and self.has_moments[k]) else None
            out.append(O.Tensor(W[k], self.R[k], m, v))
        return out

    # -- Eq. 1 ----------------------------------------------------------
    def measure(self, W, layers=None):
        """u_l for every layer (or the listed ones; others NaN) and the
        (D, A, n) sums.  In accumulate mode R then becomes W(t)."""
        u = np.full(self.nlayers, np.nan)
        sums = np.full((self.nlayers, 3), np.nan)
        for l in (range(self.nlayers) if layers is None else layers):
            d, a, n = O.layer_sums(self._tensors(l, W))
            sums[l] = (d, a, n)
            u[l] = O.update_measure(d, a, n, self.eps_w)
        if self.mode == O.ACCUMULATE and layers is None:
            self.R = [np.array(w, copy=True) for w in W]
        return u, sums

    # -- Eq. 2-4 and the staleness guard --------------------------------
    def select(self, u, tau, max_staleness, t):
        acc_before = self.delta.copy()
        tl_before = self.t_last.copy()
        mask, nsel, nonfinite = O.select_step(u, self.delta, self.t_last, tau, max_staleness, t,
                                              self.mode, self.tau_mult)
        self._undo = (acc_before, tl_before, np.asarray(u, dtype=np.float64).copy(), t)
        self.last_mask = mask
        return mask

    def adopt_decision(self, l, persist):
        """Take the other side's decision for a layer whose accumulated drift
        sits within the agreed tolerance band of the threshold."""
        acc_before, tl_before, u, t = self._undo
        acc = acc_before[l] + u[l] if self.mode == O.ACCUMULATE else u[l]
        if persist:
            self.delta[l], self.t_last[l] = 0.0, t
        else:
            self.delta[l], self.t_last[l] = acc, tl_before[l]

    def staleness(self, t):
        return O.staleness(self.t_last, self.layer_numel, t)

    # -- full layer state (§3.1) ----------------------------------------
    def layer_block_bytes(self, l):
        return O.layer_block_bytes(self._shape_tensors(l), self.align)

    def _shape_tensors(self, l):
        out = []
        for k in self.layer_tensors[l]:
            dt = np.uint16 if self.dtypes[k] == "bf16" else np.float32
            n = self.numels[k]
            m = np.zeros(n, np.float32) if self.has_moments[k] else None
            v = np.zeros(n, np.float32) if self.has_moments[k] else None
            out.append(O.Tensor(np.zeros(n, dt), None, m, v))
        return out

    def pack(self, mask, W, M, V, t):
        """Packed stream of the selected layers (ascending layer id) and the
        per-layer offsets; records a pending version per selected layer."""
        parts, offsets, off = [], np.zeros(self.nlayers, dtype=np.int64), 0
        for l in range(self.nlayers):
            offsets[l] = off
            if not mask[l]:
                continue
            block = O.pack_layer(self._tensors(l, W, M, V), self.align)
            idx = len(self.versions)
            self.versions.append(dict(layer=l, step=int(t), durable=False,
                                      digest=digest(block), nbytes=int(block.size), offset=off))
            if self.keep_blocks == "all":
                self.blocks[idx] = block
            else:
                for j in [j for j in self.blocks if self.versions[j]["layer"] == l]:
                    del self.blocks[j]
                self.blocks[idx] = block
            parts.append(block)
            off += block.size
        stream = np.concatenate(parts) if parts else np.zeros(0, np.uint8)
        return stream, offsets

    def record(self, mask, t):
        """The versions a step persists, recorded without their bytes (the
        pick of §3.5 needs only layer and step).  For long runs that check
        the composite at chosen steps only: §3.3 keeps every layer's newest
        version within the last S_max steps, so packing (pack) over the
        S_max steps before a check is enough to hold every block it picks."""
        off = 0
        for l in range(self.nlayers):
            if not mask[l]:
                continue
            nb = self._block_bytes(l)
            self.versions.append(dict(layer=l, step=int(t), durable=False, digest=None,
                                      nbytes=nb, offset=off))
            if self.keep_blocks != "all":
                for j in [j for j in self.blocks if self.versions[j]["layer"] == l]:
                    del self.blocks[j]
            off += nb

    def _block_bytes(self, l):
        cache = self.__dict__.setdefault("_block_bytes_cache", {})
        if l not in cache:
            cache[l] = int(self.layer_block_bytes(l))
        return cache[l]

    def commit(self, mask, W):
        """Snapshot mode: R_l <- W_l(t) for the persisted layers (Eq. 4 resets
        the drift reference together with the accumulator)."""
        if self.mode != O.SNAPSHOT:
            return
        for l in range(self.nlayers):
            if mask[l]:
                for k in self.layer_tensors[l]:
                    self.R[k] = np.array(W[k], copy=True)

    def mark_durable(self, t):
        for v in self.versions:
            if v["step"] == t:
                v["durable"] = True

    def drop_pending(self):
        """A crash before the copy completed: pending versions never land."""
        keep = [i for i, v in enumerate(self.versions) if v["durable"]]
        remap = {old: new for new, old in enumerate(keep)}
        self.versions = [self.versions[i] for i in keep]
        self.blocks = {remap[i]: b for i, b in self.blocks.items() if i in remap}

    # -- §3.5 / Eq. 8 ---------------------------------------------------
    def pick(self, t_fail):
        return O.composite_pick([v["layer"] for v in self.versions],
                                [v["step"] for v in self.versions],
                                [v["durable"] for v in self.versions],
                                self.nlayers, t_fail)

    def composite(self, t_fail):
        """Per tensor (w, m, v) of the composite state at t_fail."""
        pick = self.pick(t_fail)
        out = [None] * len(self.tensor_layer)
        for l in range(self.nlayers):
            if pick[l] < 0:
                raise LookupError("layer %d has no persisted version at or before step %d"
                                  % (l, t_fail))
            if int(pick[l]) not in self.blocks:
                raise LookupError("block of version %d was not kept" % pick[l])
            shape = self._shape_tensors(l)
            O.unpack_layer(self.blocks[int(pick[l])], shape, self.align)
            for k, st in zip(self.layer_tensors[l], shape):
                out[k] = (st.w, st.m, st.v)
        return out, pick
