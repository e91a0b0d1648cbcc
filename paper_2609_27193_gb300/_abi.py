"""ctypes declarations of liblayercheck.so (include/layercheck.h).

Argument marshalling only: every step of the path runs in the library's
CUDA kernels.  Loading fails loudly when the library has not been built.
"""
import ctypes as C
import os

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "liblayercheck.so")

LC_OK = 0
LC_ERR_INVALID_ARG = 1
LC_ERR_STATE = 2
LC_ERR_CUDA = 3
LC_ERR_OOM = 4
LC_ERR_CAPACITY = 5
LC_ERR_TIMEOUT = 6
LC_ERR_NOT_FOUND = 7
STATUS_NAMES = {0: "LC_OK", 1: "LC_ERR_INVALID_ARG", 2: "LC_ERR_STATE", 3: "LC_ERR_CUDA",
                4: "LC_ERR_OOM", 5: "LC_ERR_CAPACITY", 6: "LC_ERR_TIMEOUT", 7: "LC_ERR_NOT_FOUND"}

LC_BF16, LC_F32 = 0, 1
LC_DRIFT_SNAPSHOT, LC_DRIFT_ACCUMULATE = 0, 1
LC_COPY_BULK, LC_COPY_THREADS = 0, 1
LC_DEBUG_BULK_STALL = 1
LC_DEBUG_MEASURE_STALL = 2
LC_SPAN_GATHER, LC_SPAN_D2H, LC_SPAN_H2D, LC_SPAN_SCATTER = 0, 1, 2, 3
SPAN_NAMES = {0: "gather", 1: "d2h", 2: "h2d", 3: "scatter"}


class lc_segment(C.Structure):
    _fields_ = [("layer", C.c_int32), ("w_dtype", C.c_int32), ("w", C.c_void_p),
                ("snap", C.c_void_p), ("exp_avg", C.c_void_p), ("exp_avg_sq", C.c_void_p),
                ("numel", C.c_int64)]


class lc_config(C.Structure):
    _fields_ = [("eps_w", C.c_double), ("mode", C.c_int32), ("pack_align", C.c_int32),
                ("fuse_commit", C.c_int32), ("timeout_ms", C.c_int32),
                ("staging_bytes", C.c_uint64), ("copy_engine", C.c_int32),
                ("debug_flags", C.c_int32)]


class lc_select_info(C.Structure):
    _fields_ = [("step", C.c_int64), ("n_selected", C.c_int32), ("n_nonfinite", C.c_int32),
                ("bytes", C.c_uint64), ("max_staleness", C.c_int64),
                ("weighted_staleness", C.c_double)]


class lc_version(C.Structure):
    _fields_ = [("layer", C.c_int32), ("durable", C.c_int32), ("step", C.c_int64),
                ("host_ptr", C.c_void_p), ("bytes", C.c_uint64)]


class lc_optim_segment(C.Structure):
    _fields_ = [("grad", C.c_void_p), ("grad_dtype", C.c_int32), ("reserved", C.c_int32),
                ("model_copy", C.c_void_p)]


class lc_adamw_hparams(C.Structure):
    _fields_ = [("lr", C.c_double), ("beta1", C.c_double), ("beta2", C.c_double),
                ("eps", C.c_double), ("weight_decay", C.c_double)]


class lc_counters(C.Structure):
    _fields_ = [("kernel_launches", C.c_int64), ("measure_launches", C.c_int64),
                ("select_launches", C.c_int64), ("copy_launches", C.c_int64),
                ("d2h_bytes", C.c_uint64), ("h2d_bytes", C.c_uint64),
                ("bulk_copy_launches", C.c_int64), ("bulk_measure_launches", C.c_int64),
                ("measure_pool_units", C.c_int64)]


class lc_manifest_record(C.Structure):
    _fields_ = [("layer", C.c_int32), ("intact", C.c_int32), ("step", C.c_int64),
                ("offset", C.c_uint64), ("bytes", C.c_uint64), ("block_crc", C.c_uint32),
                ("layout_crc", C.c_uint32)]


class lc_store_info(C.Structure):
    _fields_ = [("arena", C.c_void_p), ("capacity", C.c_uint64), ("excluded_bytes", C.c_uint64),
                ("used_bytes", C.c_uint64), ("versions_per_layer", C.c_int32), ("reserved", C.c_int32),
                ("avoided_bytes", C.c_uint64)]


class lc_copy_span(C.Structure):
    _fields_ = [("kind", C.c_int32), ("chunk", C.c_int32), ("step", C.c_int64),
                ("bytes", C.c_uint64), ("start_ms", C.c_double), ("end_ms", C.c_double)]


ctx_p = C.c_void_p
store_p = C.c_void_p
P = C.POINTER

# name -> (restype, argtypes)
SIGNATURES = {
    "lc_config_default": (None, [P(lc_config)]),
    "lc_last_error": (C.c_char_p, []),
    "lc_create": (C.c_int, [P(ctx_p), C.c_int, C.c_void_p, P(lc_config)]),
    "lc_destroy": (None, [ctx_p]),
    "lc_register_layout": (C.c_int, [ctx_p, P(lc_segment), C.c_int32, C.c_int32, P(C.c_double)]),
    "lc_measure": (C.c_int, [ctx_p, C.c_int64]),
    "lc_layer_sums_device": (C.c_int, [ctx_p, P(C.c_void_p)]),
    "lc_set_layer_sums_buffer": (C.c_int, [ctx_p, C.c_void_p]),
    "lc_select": (C.c_int, [ctx_p, C.c_double, C.c_int32, C.c_void_p, C.c_void_p, P(C.c_uint64)]),
    "lc_last_select_info": (C.c_int, [ctx_p, P(lc_select_info)]),
    "lc_last_select_offsets": (C.c_int, [ctx_p, C.c_void_p]),
    "lc_pack_device": (C.c_int, [ctx_p, C.c_void_p, C.c_uint64]),
    "lc_pack_async": (C.c_int, [ctx_p, store_p]),
    "lc_commit_snapshot": (C.c_int, [ctx_p]),
    "lc_wait_durable": (C.c_int, [ctx_p, C.c_int64, C.c_int32]),
    "lc_restore": (C.c_int, [ctx_p, store_p, C.c_int64, C.c_void_p]),
    "lc_layer_block_bytes": (C.c_int, [ctx_p, C.c_int32, P(C.c_uint64)]),
    "lc_get_counters": (C.c_int, [ctx_p, P(lc_counters)]),
    "lc_store_create": (C.c_int, [P(store_p), ctx_p, C.c_uint64, C.c_int32]),
    "lc_store_destroy": (None, [store_p]),
    "lc_store_clear": (C.c_int, [store_p]),
    "lc_store_num_versions": (C.c_int64, [store_p]),
    "lc_store_get_version": (C.c_int, [store_p, C.c_int64, P(lc_version)]),
    "lc_store_plan": (C.c_int, [store_p, C.c_int64, C.c_void_p]),
    "lc_store_exclude": (C.c_int, [store_p, C.c_uint64, C.c_uint64]),
    "lc_store_get_info": (C.c_int, [store_p, P(lc_store_info)]),
    "lc_store_check_dma": (C.c_int, [store_p, ctx_p, C.c_uint64, C.c_int32, C.c_double, C.c_void_p,
                                     C.c_int64, P(C.c_uint64)]),
    "lc_step_async": (C.c_int, [ctx_p, C.c_int64, C.c_double, C.c_int32, C.c_void_p, C.c_uint64]),
    "lc_step_wait": (C.c_int, [ctx_p, C.c_int64, C.c_int32, C.c_void_p, C.c_void_p, P(C.c_uint64)]),
    "lc_step_graph_create": (C.c_int, [ctx_p, C.c_double, C.c_int32, C.c_void_p, C.c_uint64]),
    "lc_step_graph_launch": (C.c_int, [ctx_p, P(C.c_int64)]),
    "lc_register_optimizer": (C.c_int, [ctx_p, P(lc_optim_segment), C.c_int32]),
    "lc_adamw_step_measure": (C.c_int, [ctx_p, C.c_int64, P(lc_adamw_hparams)]),
    "lc_measure_noalloc": (C.c_int, [C.c_int, C.c_void_p, P(lc_segment), C.c_int32, C.c_int32,
                                     C.c_void_p]),
    "lc_copy_trace_enable": (C.c_int, [ctx_p, C.c_int32]),
    "lc_copy_trace_read": (C.c_int, [ctx_p, P(lc_copy_span), C.c_int64, P(C.c_int64), P(C.c_int64)]),
    "lc_crc32c": (C.c_uint32, [C.c_void_p, C.c_uint64, C.c_uint32]),
    "lc_store_persist_dir": (C.c_int, [store_p, C.c_char_p, C.c_int32, P(C.c_uint64)]),
    "lc_store_load_dir": (C.c_int, [ctx_p, C.c_char_p, C.c_int64, P(store_p), C.c_void_p]),
    "lc_manifest_read": (C.c_int, [C.c_char_p, C.c_int32, P(lc_manifest_record), C.c_int64,
                                   P(C.c_int64), P(C.c_int32), P(C.c_uint32), P(C.c_int32)]),
}

# limits of lc_measure_noalloc (include/layercheck.h)
LC_NOALLOC_MAX_SEGMENTS = 512
LC_NOALLOC_MAX_LAYERS = 512
LC_NOALLOC_SCRATCH_BYTES = 192 * 1024

_lib = None


def load():
    """The loaded library; raises if it was never built (no fallback)."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise ImportError("liblayercheck.so is not built (run __graft_entry__.build() or "
                              "python paper_2609_27193_gb300/build.py); there is no CPU fallback")
        lib = C.CDLL(LIB_PATH)
        for name, (res, args) in SIGNATURES.items():
            fn = getattr(lib, name)
            fn.restype = res
            fn.argtypes = args
        _lib = lib
    return _lib


class LCError(RuntimeError):
    def __init__(self, status, msg):
        super().__init__("%s: %s" % (STATUS_NAMES.get(status, status), msg))
        self.status = status


def check(status):
    if status != LC_OK:
        raise LCError(status, load().lc_last_error().decode(errors="replace"))
    return status
