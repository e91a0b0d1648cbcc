"""GB300-native LayerCheck hot path: Python binding of liblayercheck.so.

LayerCheck (adaptive layer-wise checkpointing) measures at every checkpoint
opportunity how far each layer's weights drifted (§3.2 Eq. 1), persists the
layers whose accumulated drift reached a threshold or whose staleness
reached S_max (§3.2 Eq. 2-4, §3.3) together with their Adam moments (§3.1),
and restores the mixed-timestamp composite of the latest persisted versions
(§3.5, Eq. 8).  Every step runs in the CUDA kernels of liblayercheck.so;
this module only marshals torch tensors, streams and numpy arrays into the
C ABI of include/layercheck.h (the raw functions keep their C names in
``paper_2609_27193_gb300._abi``).  There is no CPU fallback.
"""
import ctypes as C
import os

import numpy as np

from . import _abi
from ._abi import (LC_BF16, LC_COPY_BULK, LC_COPY_THREADS, LC_DEBUG_BULK_STALL, LC_DEBUG_MEASURE_STALL,
                   LC_DRIFT_ACCUMULATE, LC_DRIFT_SNAPSHOT, LC_F32, LCError, check, lc_config,
                   lc_counters, lc_segment, lc_select_info, lc_version)

__all__ = ["LayerCheck", "Store", "LCError", "LC_BF16", "LC_F32", "LC_DRIFT_SNAPSHOT",
           "LC_DRIFT_ACCUMULATE", "LC_DEBUG_BULK_STALL", "LC_DEBUG_MEASURE_STALL", "library", "segment",
           "crc32c",
           "manifest_read"]


def library():
    """The loaded ctypes library (raises ImportError when not built)."""
    return _abi.load()


def crc32c(data, crc=0):
    """CRC-32C of a bytes-like object or contiguous numpy array (host)."""
    buf = np.ascontiguousarray(np.frombuffer(data, dtype=np.uint8) if not isinstance(data, np.ndarray)
                               else data.view(np.uint8).reshape(-1))
    return int(library().lc_crc32c(buf.ctypes.data, buf.size, int(crc)))


def manifest_read(path, verify_blocks=True):
    """The valid records of a checkpoint directory's manifest (no GPU):
    (records as dicts in file order, nlayers, layout CRC, torn tail?)."""
    from ._abi import lc_manifest_record
    lib = library()
    n = C.c_int64(0)
    nl = C.c_int32(0)
    lay = C.c_uint32(0)
    torn = C.c_int32(0)
    check(lib.lc_manifest_read(os.fsencode(path), 0, None, 0, C.byref(n), C.byref(nl), C.byref(lay),
                               C.byref(torn)))
    recs = (lc_manifest_record * max(1, n.value))()
    check(lib.lc_manifest_read(os.fsencode(path), int(bool(verify_blocks)), recs, n.value, C.byref(n),
                               C.byref(nl), C.byref(lay), C.byref(torn)))
    out = [{name: getattr(recs[i], name) for name, _ in lc_manifest_record._fields_}
           for i in range(n.value)]
    return out, nl.value, lay.value, bool(torn.value)


def _dtype_code(t):
    import torch
    if t.dtype == torch.bfloat16:
        return LC_BF16
    if t.dtype == torch.float32:
        return LC_F32
    raise TypeError("weights must be bfloat16 or float32, got %s" % t.dtype)


def segment(layer, w, snap, exp_avg=None, exp_avg_sq=None):
    """An lc_segment over torch CUDA tensors (contiguous, same numel); snap
    may be None in accumulate mode (fused optimizer path only).  The library
    keeps raw pointers, so the segment holds references to the tensors and
    the context that registers it keeps the segment."""
    import torch
    for name, t in (("w", w), ("snap", snap), ("exp_avg", exp_avg), ("exp_avg_sq", exp_avg_sq)):
        if t is not None and not t.is_contiguous():
            raise ValueError("%s must be contiguous" % name)
        if t is not None and t.device != w.device:
            raise ValueError("%s must be on the device of w" % name)
    if snap is not None and (snap.dtype != w.dtype or snap.numel() != w.numel()):
        raise ValueError("snap must match w in dtype and size")
    if (exp_avg is None) != (exp_avg_sq is None):
        raise ValueError("exp_avg and exp_avg_sq must both be given or both be None")
    for name, t in (("exp_avg", exp_avg), ("exp_avg_sq", exp_avg_sq)):
        if t is not None and (t.dtype != torch.float32 or t.numel() != w.numel()):
            raise ValueError("%s must be float32 with the numel of w" % name)
    s = lc_segment(int(layer), _dtype_code(w), w.data_ptr(),
                   snap.data_ptr() if snap is not None else None,
                   exp_avg.data_ptr() if exp_avg is not None else None,
                   exp_avg_sq.data_ptr() if exp_avg_sq is not None else None,
                   int(w.numel()))
    s._refs = (w, snap, exp_avg, exp_avg_sq)
    return s


class LayerCheck:
    """One library context on one device and one CUDA stream."""

    def __init__(self, device=0, stream=None, eps_w=1e-8, mode=LC_DRIFT_SNAPSHOT,
                 pack_align=256, fuse_commit=True, timeout_ms=60000, staging_bytes=512 << 20,
                 copy_engine="bulk", debug_flags=0):
        lib = library()
        cfg = lc_config()
        lib.lc_config_default(C.byref(cfg))
        cfg.eps_w, cfg.mode, cfg.pack_align = float(eps_w), int(mode), int(pack_align)
        cfg.fuse_commit, cfg.timeout_ms = int(bool(fuse_commit)), int(timeout_ms)
        cfg.staging_bytes = int(staging_bytes)
        engines = {"bulk": LC_COPY_BULK, "threads": LC_COPY_THREADS}
        if copy_engine not in engines:
            raise ValueError("copy_engine must be one of %s" % sorted(engines))
        cfg.copy_engine = engines[copy_engine]
        cfg.debug_flags = int(debug_flags)
        if stream is None:
            import torch
            stream = torch.cuda.current_stream(device)
        self.stream = stream
        handle = stream.cuda_stream if hasattr(stream, "cuda_stream") else int(stream or 0)
        ctx = C.c_void_p()
        check(lib.lc_create(C.byref(ctx), int(device), C.c_void_p(handle), C.byref(cfg)))
        self._lib, self._ctx = lib, ctx
        self.device = int(device)
        self.nlayers = 0
        self._keep = []

    # -- lifecycle -----------------------------------------------------
    def close(self):
        if getattr(self, "_ctx", None) and self._ctx.value:
            self._lib.lc_destroy(self._ctx)
            self._ctx = C.c_void_p()

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def __enter__(self):
        return self

    def __exit__(self, *exc):
        self.close()

    @property
    def handle(self):
        return self._ctx

    # -- the path ------------------------------------------------------
    def register_layout(self, segments, nlayers, tau_mult=None):
        arr = (lc_segment * len(segments))(*segments)
        mult = None
        if tau_mult is not None:
            m = np.ascontiguousarray(tau_mult, dtype=np.float64)
            mult = m.ctypes.data_as(C.POINTER(C.c_double))
            self._keep.append(m)
        check(self._lib.lc_register_layout(self._ctx, arr, len(segments), int(nlayers), mult))
        self.nlayers = int(nlayers)
        self._numels = [int(sg.numel) for sg in segments]
        self._keep.append([getattr(sg, "_refs", None) for sg in segments])

    def measure(self, step):
        check(self._lib.lc_measure(self._ctx, int(step)))

    def register_optimizer(self, grads, model_copies=None):
        """Gradients (and optional bf16 model copies) of every segment, in the
        order of register_layout, for the fused AdamW + drift step."""
        import torch
        from ._abi import lc_optim_segment
        n = len(grads)
        numels = getattr(self, "_numels", [])
        if n != len(numels) or (model_copies is not None and len(model_copies) != n):
            raise ValueError("need one gradient (and model copy) per registered segment")
        arr = (lc_optim_segment * n)()
        for i, g in enumerate(grads):
            mc = None if model_copies is None else model_copies[i]
            if not g.is_contiguous() or g.numel() != numels[i]:
                raise ValueError("gradient %d must be contiguous with the numel of its segment" % i)
            if mc is not None and (mc.dtype != torch.bfloat16 or not mc.is_contiguous()
                                   or mc.numel() != numels[i]):
                raise ValueError("model copy %d must be contiguous bfloat16 with the numel of its segment" % i)
            arr[i] = lc_optim_segment(g.data_ptr(), _dtype_code(g), 0,
                                      mc.data_ptr() if mc is not None else None)
        self._keep.append((grads, model_copies))
        check(self._lib.lc_register_optimizer(self._ctx, arr, n))

    def adamw_step_measure(self, step, lr, beta1=0.9, beta2=0.999, eps=1e-8, weight_decay=0.0):
        """One fused AdamW step on every segment with the Eq. 1 sums of the
        update (takes the place of measure)."""
        from ._abi import lc_adamw_hparams
        hp = lc_adamw_hparams(float(lr), float(beta1), float(beta2), float(eps), float(weight_decay))
        check(self._lib.lc_adamw_step_measure(self._ctx, int(step), C.byref(hp)))

    def layer_sums_ptr(self):
        p = C.c_void_p()
        check(self._lib.lc_layer_sums_device(self._ctx, C.byref(p)))
        return p.value

    def set_layer_sums_buffer(self, tensor):
        """Keep the (D, A, n) sums in a caller-owned float64 CUDA tensor of
        3*nlayers elements (all-reduce it between measure and select)."""
        import torch
        if tensor.dtype != torch.float64 or tensor.numel() != 3 * self.nlayers or not tensor.is_cuda:
            raise ValueError("need a float64 CUDA tensor of 3*nlayers elements")
        self._keep.append(tensor)
        check(self._lib.lc_set_layer_sums_buffer(self._ctx, C.c_void_p(tensor.data_ptr())))

    def select(self, tau, max_staleness):
        """Decision of this step: (mask uint8[N], u float64[N], packed bytes)."""
        mask = np.zeros(self.nlayers, dtype=np.uint8)
        u = np.zeros(self.nlayers, dtype=np.float64)
        nbytes = C.c_uint64(0)
        check(self._lib.lc_select(self._ctx, float(tau), int(max_staleness), mask.ctypes.data,
                                  u.ctypes.data, C.byref(nbytes)))
        return mask, u, nbytes.value

    def info(self):
        i = lc_select_info()
        check(self._lib.lc_last_select_info(self._ctx, C.byref(i)))
        return dict(step=i.step, n_selected=i.n_selected, n_nonfinite=i.n_nonfinite,
                    bytes=i.bytes, max_staleness=i.max_staleness,
                    weighted_staleness=i.weighted_staleness)

    def offsets(self):
        o = np.zeros(self.nlayers, dtype=np.uint64)
        check(self._lib.lc_last_select_offsets(self._ctx, o.ctypes.data))
        return o

    def step_async(self, step, tau, max_staleness, dst):
        """Enqueue a whole step (measure, select, pack into dst, commit) with
        no host round trip; read the decision later with step_wait."""
        check(self._lib.lc_step_async(self._ctx, int(step), float(tau), int(max_staleness),
                                      C.c_void_p(dst.data_ptr()), int(dst.numel() * dst.element_size())))

    def step_wait(self, step, timeout_ms=0):
        """Decision of an asynchronous or graph step: (mask, u, bytes)."""
        mask = np.zeros(self.nlayers, dtype=np.uint8)
        u = np.zeros(self.nlayers, dtype=np.float64)
        nbytes = C.c_uint64(0)
        check(self._lib.lc_step_wait(self._ctx, int(step), int(timeout_ms), mask.ctypes.data,
                                     u.ctypes.data, C.byref(nbytes)))
        return mask, u, nbytes.value

    def step_graph_create(self, tau, max_staleness, dst):
        """Capture one step (fixed tau, S_max and destination) as a CUDA graph."""
        self._keep.append(dst)
        check(self._lib.lc_step_graph_create(self._ctx, float(tau), int(max_staleness),
                                             C.c_void_p(dst.data_ptr()),
                                             int(dst.numel() * dst.element_size())))

    def step_graph_launch(self):
        """Replay the captured step; returns its step number."""
        s = C.c_int64(0)
        check(self._lib.lc_step_graph_launch(self._ctx, C.byref(s)))
        return s.value

    def pack_device(self, dst):
        """Gather into a uint8 CUDA (or pinned host) tensor."""
        check(self._lib.lc_pack_device(self._ctx, C.c_void_p(dst.data_ptr()),
                                       int(dst.numel() * dst.element_size())))

    def pack_async(self, store):
        check(self._lib.lc_pack_async(self._ctx, store.handle))

    def commit_snapshot(self):
        check(self._lib.lc_commit_snapshot(self._ctx))

    def wait_durable(self, step, timeout_ms=0):
        check(self._lib.lc_wait_durable(self._ctx, int(step), int(timeout_ms)))

    def restore(self, store, t_fail):
        steps = np.zeros(self.nlayers, dtype=np.int64)
        check(self._lib.lc_restore(self._ctx, store.handle, int(t_fail), steps.ctypes.data))
        return steps

    def load_dir(self, path, t_fail):
        """§3.5 recovery from a checkpoint directory: each layer's newest
        intact version at or before t_fail, read into a new Store (one
        version per layer) for restore().  Returns (store, steps)."""
        steps = np.zeros(self.nlayers, dtype=np.int64)
        h = C.c_void_p()
        check(self._lib.lc_store_load_dir(self._ctx, os.fsencode(path), int(t_fail), C.byref(h),
                                          steps.ctypes.data))
        return Store._adopt(h, self.nlayers), steps

    def layer_block_bytes(self, layer):
        b = C.c_uint64(0)
        check(self._lib.lc_layer_block_bytes(self._ctx, int(layer), C.byref(b)))
        return b.value

    def trace_copies(self, enable=True):
        """Start (or stop) timing the staged host copies of pack_async and
        restore chunk by chunk; clears the previous record."""
        check(self._lib.lc_copy_trace_enable(self._ctx, int(bool(enable))))

    def copy_trace(self):
        """The recorded spans as a list of dicts (kind, chunk, step, bytes,
        start_ms, end_ms), in record order, and the number dropped."""
        from ._abi import SPAN_NAMES, lc_copy_span
        n = C.c_int64(0)
        dropped = C.c_int64(0)
        check(self._lib.lc_copy_trace_read(self._ctx, None, 0, C.byref(n), C.byref(dropped)))
        arr = (lc_copy_span * max(1, n.value))()
        check(self._lib.lc_copy_trace_read(self._ctx, arr, n.value, C.byref(n), C.byref(dropped)))
        out = [dict(kind=SPAN_NAMES.get(arr[i].kind, arr[i].kind), chunk=arr[i].chunk, step=arr[i].step,
                    bytes=arr[i].bytes, start_ms=arr[i].start_ms, end_ms=arr[i].end_ms)
               for i in range(n.value)]
        return out, dropped.value

    def counters(self):
        c = lc_counters()
        check(self._lib.lc_get_counters(self._ctx, C.byref(c)))
        return {name: getattr(c, name) for name, _ in lc_counters._fields_}


class Store:
    """Pinned-host store of persisted layer versions (library-owned memory)."""

    def __init__(self, lc, capacity_bytes=0, versions_per_layer=0):
        self._lib = library()
        h = C.c_void_p()
        check(self._lib.lc_store_create(C.byref(h), lc.handle, int(capacity_bytes),
                                        int(versions_per_layer)))
        self._h = h
        self.nlayers = lc.nlayers

    @classmethod
    def _adopt(cls, handle, nlayers):
        st = cls.__new__(cls)
        st._lib, st._h, st.nlayers = library(), handle, nlayers
        return st

    @property
    def handle(self):
        return self._h

    def persist_dir(self, path, sync=False):
        """Appends the durable versions the directory does not hold yet
        (file tier, format in layercheck.h); returns the block bytes written."""
        n = C.c_uint64(0)
        check(self._lib.lc_store_persist_dir(self._h, os.fsencode(path), int(bool(sync)), C.byref(n)))
        return n.value

    def close(self):
        if getattr(self, "_h", None) and self._h.value:
            self._lib.lc_store_destroy(self._h)
            self._h = C.c_void_p()

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def clear(self):
        check(self._lib.lc_store_clear(self._h))

    def __len__(self):
        return int(self._lib.lc_store_num_versions(self._h))

    def version(self, i):
        v = lc_version()
        check(self._lib.lc_store_get_version(self._h, int(i), C.byref(v)))
        return dict(layer=v.layer, durable=bool(v.durable), step=v.step, host_ptr=v.host_ptr,
                    bytes=v.bytes)

    def versions(self):
        return [self.version(i) for i in range(len(self))]

    def block(self, i):
        """The packed block of version i as a numpy uint8 view (no copy)."""
        v = self.version(i)
        if v["bytes"] == 0:
            return np.zeros(0, np.uint8)
        buf = (C.c_uint8 * v["bytes"]).from_address(v["host_ptr"])
        return np.frombuffer(buf, dtype=np.uint8)

    def info(self):
        """Arena base address, capacity, excluded and used bytes."""
        from ._abi import lc_store_info
        i = lc_store_info()
        check(self._lib.lc_store_get_info(self._h, C.byref(i)))
        return dict(arena=i.arena, capacity=i.capacity, excluded_bytes=i.excluded_bytes,
                    used_bytes=i.used_bytes, versions_per_layer=i.versions_per_layer,
                    avoided_bytes=i.avoided_bytes)

    @property
    def capacity(self):
        return self.info()["capacity"]

    def exclude(self, offset, nbytes):
        """Keep bytes [offset, offset + nbytes) of the arena out of use."""
        check(self._lib.lc_store_exclude(self._h, int(offset), int(nbytes)))

    def check_dma(self, lc, region_bytes=256 << 20, min_fraction=0.5, passes=4):
        """Time `passes` device->host copies into every region of the (empty)
        arena and exclude the regions whose slowest pass ran below
        min_fraction x the median of the regions' fastest passes, slowest
        first, as long as a step that persists every layer still fits.
        Returns (each region's slowest GB/s as a numpy array, excluded
        bytes)."""
        cap = int(self.capacity)
        n = -(-cap // int(region_bytes))
        rates = np.zeros(n, dtype=np.float64)
        ex = C.c_uint64(0)
        check(self._lib.lc_store_check_dma(self._h, lc.handle, int(region_bytes), int(passes),
                                           float(min_fraction), rates.ctypes.data, n, C.byref(ex)))
        return rates, ex.value

    def plan(self, t_fail):
        pick = np.zeros(self.nlayers, dtype=np.int64)
        check(self._lib.lc_store_plan(self._h, int(t_fail), pick.ctypes.data))
        return pick
