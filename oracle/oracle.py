"""ctypes wrapper of the C oracle (TEST INFRASTRUCTURE ONLY).

Arrays are numpy: bf16 tensors are carried as their uint16 bit patterns,
fp32 tensors as float32.  Every function here only marshals arguments for
the C restatement in lc_oracle.c, which cites the paper passage it follows.
"""
import ctypes as C
import os

import numpy as np

from .build import build_oracle

BF16, F32 = 0, 1
SNAPSHOT, ACCUMULATE = 0, 1

_lib = None


class AdamW(C.Structure):
    _fields_ = [("lr", C.c_double), ("beta1", C.c_double), ("beta2", C.c_double),
                ("eps", C.c_double), ("weight_decay", C.c_double)]


class _Tensor(C.Structure):
    _fields_ = [("w", C.c_void_p), ("r", C.c_void_p), ("m", C.c_void_p),
                ("v", C.c_void_p), ("numel", C.c_int64), ("dtype", C.c_int32),
                ("reserved", C.c_int32)]


def lib():
    global _lib
    if _lib is None:
        _lib = declare(C.CDLL(build_oracle()))
    return _lib


def declare(L):
    """Sets the ctypes signatures of an oracle library and returns it."""
    L.lco_bf16_value.restype = C.c_double
    L.lco_bf16_value.argtypes = [C.c_uint16]
    L.lco_layer_sums.restype = None
    L.lco_layer_sums.argtypes = [C.POINTER(_Tensor), C.c_int32, C.POINTER(C.c_double)]
    L.lco_update_measure.restype = C.c_double
    L.lco_update_measure.argtypes = [C.c_double] * 4
    L.lco_select_step.restype = C.c_int32
    L.lco_select_step.argtypes = [C.c_int32, C.c_void_p, C.c_void_p, C.c_void_p,
                                  C.c_void_p, C.c_double, C.c_int32, C.c_int64,
                                  C.c_int32, C.c_void_p, C.POINTER(C.c_int32)]
    L.lco_staleness.restype = None
    L.lco_staleness.argtypes = [C.c_int32, C.c_void_p, C.c_void_p, C.c_int64,
                                C.POINTER(C.c_int64), C.POINTER(C.c_double)]
    L.lco_layer_block_bytes.restype = C.c_uint64
    L.lco_layer_block_bytes.argtypes = [C.POINTER(_Tensor), C.c_int32, C.c_uint32]
    L.lco_pack_layer.restype = C.c_uint64
    L.lco_pack_layer.argtypes = [C.POINTER(_Tensor), C.c_int32, C.c_uint32, C.c_void_p]
    L.lco_unpack_layer.restype = C.c_int32
    L.lco_unpack_layer.argtypes = [C.c_void_p, C.c_uint64, C.POINTER(_Tensor),
                                   C.c_int32, C.c_uint32]
    L.lco_adamw_constants.restype = None
    L.lco_adamw_constants.argtypes = [C.POINTER(AdamW), C.c_int64, C.POINTER(C.c_float)]
    L.lco_bf16_round.restype = C.c_uint16
    L.lco_bf16_round.argtypes = [C.c_float]
    L.lco_adamw_step.restype = None
    L.lco_adamw_step.argtypes = [C.POINTER(AdamW), C.c_int64, C.c_int64, C.c_void_p, C.c_void_p,
                                 C.c_void_p, C.c_void_p, C.c_int32, C.c_void_p,
                                 C.POINTER(C.c_double), C.POINTER(C.c_double)]
    L.lco_composite_pick.restype = None
    L.lco_composite_pick.argtypes = [C.c_int32, C.c_void_p, C.c_void_p, C.c_void_p,
                                     C.c_int32, C.c_int64, C.c_void_p]
    return L


class Tensor:
    """One parameter tensor of a layer: w, r (uint16 bf16 bits or float32),
    m, v (float32 or None).  Arrays must be C-contiguous and 1-D."""

    def __init__(self, w, r=None, m=None, v=None):
        self.w = np.ascontiguousarray(w)
        self.r = np.ascontiguousarray(r) if r is not None else None
        self.m = np.ascontiguousarray(m, dtype=np.float32) if m is not None else None
        self.v = np.ascontiguousarray(v, dtype=np.float32) if v is not None else None
        if self.w.dtype == np.uint16:
            self.dtype = BF16
        elif self.w.dtype == np.float32:
            self.dtype = F32
        else:
            raise TypeError("weights must be uint16 (bf16 bits) or float32")
        if self.r is not None and self.r.dtype != self.w.dtype:
            raise TypeError("reference and weights must share a dtype")
        self.numel = int(self.w.size)
        for a in (self.r, self.m, self.v):
            if a is not None and a.size != self.numel:
                raise ValueError("tensor arrays differ in length")


def _ptr(a):
    return None if a is None else a.ctypes.data


def _structs(tensors):
    arr = (_Tensor * max(1, len(tensors)))()
    for i, t in enumerate(tensors):
        arr[i] = _Tensor(_ptr(t.w), _ptr(t.r), _ptr(t.m), _ptr(t.v), t.numel, t.dtype, 0)
    return arr


def bf16_value(bits):
    return lib().lco_bf16_value(int(bits))


def layer_sums(tensors):
    """(D, A, n) of Eq. 1 for one layer given as a list of Tensor."""
    out = (C.c_double * 3)()
    lib().lco_layer_sums(_structs(tensors), len(tensors), out)
    return out[0], out[1], out[2]


def update_measure(d_sum, a_sum, n, eps_w):
    return lib().lco_update_measure(d_sum, a_sum, n, eps_w)


def select_step(u, delta, t_last, tau, max_staleness, t, mode=SNAPSHOT, tau_mult=None):
    """Mutates delta (float64) and t_last (int64) in place; returns
    (mask uint8, n_selected, n_nonfinite)."""
    u = np.ascontiguousarray(u, dtype=np.float64)
    assert delta.dtype == np.float64 and t_last.dtype == np.int64
    assert delta.flags.c_contiguous and t_last.flags.c_contiguous
    n = u.size
    mult = None if tau_mult is None else np.ascontiguousarray(tau_mult, dtype=np.float64)
    mask = np.zeros(n, dtype=np.uint8)
    nf = C.c_int32(0)
    nsel = lib().lco_select_step(n, _ptr(u), _ptr(delta), _ptr(t_last), _ptr(mult),
                                 float(tau), int(max_staleness), int(t), int(mode),
                                 _ptr(mask), C.byref(nf))
    if nsel < 0:
        raise ValueError("oracle select rejected its arguments")
    return mask, nsel, nf.value


def staleness(t_last, layer_numel, t):
    t_last = np.ascontiguousarray(t_last, dtype=np.int64)
    numel = np.ascontiguousarray(layer_numel, dtype=np.int64)
    mx, wt = C.c_int64(0), C.c_double(0)
    lib().lco_staleness(t_last.size, _ptr(t_last), _ptr(numel), int(t), C.byref(mx), C.byref(wt))
    return mx.value, wt.value


def layer_block_bytes(tensors, align=256):
    return int(lib().lco_layer_block_bytes(_structs(tensors), len(tensors), align))


def pack_layer(tensors, align=256):
    n = layer_block_bytes(tensors, align)
    dst = np.empty(n, dtype=np.uint8)
    got = lib().lco_pack_layer(_structs(tensors), len(tensors), align, _ptr(dst))
    assert got == n
    return dst


def unpack_layer(block, tensors, align=256):
    """Writes w, m, v of `tensors` (which must own writable arrays)."""
    block = np.ascontiguousarray(block, dtype=np.uint8)
    rc = lib().lco_unpack_layer(_ptr(block), block.size, _structs(tensors), len(tensors), align)
    if rc != 0:
        raise ValueError("block does not match the layer layout or has non-zero padding")


def composite_pick(v_layer, v_step, v_durable, nlayers, t_fail):
    v_layer = np.ascontiguousarray(v_layer, dtype=np.int32)
    v_step = np.ascontiguousarray(v_step, dtype=np.int64)
    v_durable = np.ascontiguousarray(v_durable, dtype=np.uint8)
    pick = np.empty(nlayers, dtype=np.int64)
    lib().lco_composite_pick(v_layer.size, _ptr(v_layer), _ptr(v_step), _ptr(v_durable),
                             nlayers, int(t_fail), _ptr(pick))
    return pick


def adamw_constants(hp, t):
    out = (C.c_float * 9)()
    lib().lco_adamw_constants(C.byref(AdamW(*hp)), int(t), out)
    return list(out)


def bf16_round(f):
    return int(lib().lco_bf16_round(float(f)))


def adamw_step(hp, t, p, m, v, grad, model=None):
    """One AdamW step in place on float32 arrays p, m, v; grad is uint16
    (bf16 bits) or float32; model (uint16, nullable) receives bf16(p).
    Returns (D, A) of Eq. 1 for the update.  hp = (lr, beta1, beta2, eps, wd)."""
    for a in (p, m, v):
        assert a.dtype == np.float32 and a.flags.c_contiguous
    grad = np.ascontiguousarray(grad)
    is_bf16 = grad.dtype == np.uint16
    assert is_bf16 or grad.dtype == np.float32
    if model is not None:
        assert model.dtype == np.uint16 and model.flags.c_contiguous
    d, a = C.c_double(0), C.c_double(0)
    lib().lco_adamw_step(C.byref(AdamW(*hp)), int(t), p.size, _ptr(p), _ptr(m), _ptr(v),
                         _ptr(grad), int(is_bf16), _ptr(model), C.byref(d), C.byref(a))
    return d.value, a.value
