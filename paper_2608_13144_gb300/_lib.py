"""ctypes declarations of the C ABI in include/lipcache.h.

Loading fails loudly when liblipcache.so is missing: there is no CPU or
PyTorch fallback for any step of the lookup.
"""
from __future__ import annotations

import ctypes as C
import os

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "liblipcache.so")

OK, E_INVALID, E_STATE, E_DEGENERATE_HEAD, E_FULL, E_NOT_CONVERGED, E_CUDA, E_NOMEM, E_DEVICE = range(9)
STATUS_NAMES = {0: "OK", 1: "E_INVALID", 2: "E_STATE", 3: "E_DEGENERATE_HEAD", 4: "E_FULL", 5: "E_NOT_CONVERGED",
                6: "E_CUDA", 7: "E_NOMEM", 8: "E_DEVICE"}
RADIUS_CONSERVATIVE, RADIUS_TIGHT = 0, 1
NOALLOC_SCRATCH_BYTES = 4259840  # LIPCACHE_NOALLOC_SCRATCH_BYTES
PROBE_AUTO, PROBE_TENSOR, PROBE_EXACT, PROBE_TENSOR_SINGLE, PROBE_TENSOR_PAIR = 0, 1, 2, 3, 4

# Every symbol the header declares; tests check the library exports them all.
EXPORTS = ["lipcache_create", "lipcache_set_head", "lipcache_insert", "lipcache_probe", "lipcache_probe_host",
           "lipcache_probe_noalloc", "lipcache_probe_writeback", "lipcache_consistency",
           "lipcache_set_radius_policy", "lipcache_insert_select", "lipcache_set_debug", "lipcache_read_entries", "lipcache_read_head",
           "lipcache_set_probe_path", "lipcache_set_radius_scale", "lipcache_set_spectral_options",
           "lipcache_reserve", "lipcache_enable_timing", "lipcache_get_info", "lipcache_reset_stats",
           "lipcache_size", "lipcache_destroy", "lipcache_last_error"]


class Info(C.Structure):
    _fields_ = [("d", C.c_int32), ("C", C.c_int32), ("d_pad", C.c_int32), ("radius_mode", C.c_int32),
                ("capacity", C.c_int64), ("size", C.c_int64), ("head_set", C.c_int32),
                ("sigma_iterations", C.c_int32), ("sigma", C.c_double), ("sigma_residual", C.c_double),
                ("radius_scale", C.c_double), ("eps_recheck", C.c_double), ("c_screen", C.c_double),
                ("candidates", C.c_int64), ("device_errors", C.c_int64), ("probe_path", C.c_int32),
                ("last_probe_path", C.c_int32), ("last_probe_ms", C.c_float), ("num_sms", C.c_int32),
                ("kernel_ms_total", C.c_double), ("kernel_launches", C.c_int64), ("last_grid", C.c_int32),
                ("last_cluster", C.c_int32), ("radius_policy", C.c_int32), ("last_insert_kernel", C.c_int32),
                ("policy_param", C.c_double), ("insert_kernel_ms_total", C.c_double),
                ("insert_kernel_launches", C.c_int64), ("insert_refined_pairs", C.c_int64),
                ("insert_full_rows", C.c_int64), ("insert_fp64_rows", C.c_int64)]


class LipCacheError(RuntimeError):
    def __init__(self, status: int, message: str):
        super().__init__(f"{STATUS_NAMES.get(status, status)}: {message}")
        self.status = status


_lib = None


def load(path: str = LIB_PATH):
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(path):
        raise ImportError(f"{path} is missing: build it with paper_2608_13144_gb300.build.build() "
                          "(there is no fallback implementation)")
    L = C.CDLL(path)
    vp, i32, i64, f64 = C.c_void_p, C.c_int32, C.c_int64, C.c_double
    sig = {
        "lipcache_create": ([i32, i32, i64, i32, C.POINTER(vp)], C.c_int),
        "lipcache_set_head": ([vp, vp, vp, C.POINTER(f64), vp], C.c_int),
        "lipcache_insert": ([vp, vp, i64, vp, i32, vp, vp, C.POINTER(i64), vp], C.c_int),
        "lipcache_probe": ([vp, vp, i64, vp, vp, vp, vp], C.c_int),
        "lipcache_probe_host": ([vp, vp, i64, vp, vp, vp, vp], C.c_int),
        "lipcache_probe_noalloc": ([vp, vp, i64, vp, vp, vp, vp], C.c_int),
        "lipcache_probe_writeback": ([vp, vp, i64, vp, i32, vp, vp, vp, vp, C.POINTER(i64), vp], C.c_int),
        "lipcache_consistency": ([vp, vp, i64, vp, vp, C.POINTER(i64), C.POINTER(i64), vp], C.c_int),
        "lipcache_set_radius_policy": ([vp, i32, f64, vp, vp], C.c_int),
        "lipcache_insert_select": ([vp, vp, i64, vp, i32, i32, i64, i32, vp, vp, C.POINTER(i64), vp], C.c_int),
        "lipcache_set_debug": ([vp, i32], C.c_int),
        "lipcache_read_entries": ([vp, i64, i64, vp, vp, vp, vp, vp], C.c_int),
        "lipcache_read_head": ([vp, vp, vp, vp], C.c_int),
        "lipcache_set_probe_path": ([vp, i32], C.c_int),
        "lipcache_set_radius_scale": ([vp, f64], C.c_int),
        "lipcache_set_spectral_options": ([vp, i32, i32], C.c_int),
        "lipcache_reserve": ([vp, i64], C.c_int),
        "lipcache_enable_timing": ([vp, i32], C.c_int),
        "lipcache_get_info": ([vp, C.POINTER(Info)], C.c_int),
        "lipcache_reset_stats": ([vp], C.c_int),
        "lipcache_size": ([vp], i64),
        "lipcache_destroy": ([vp], None),
        "lipcache_last_error": ([], C.c_char_p),
    }
    for name, (args, res) in sig.items():
        fn = getattr(L, name)
        fn.argtypes = args
        fn.restype = res
    _lib = L
    return L


def check(status: int) -> None:
    if status != OK:
        msg = load().lipcache_last_error()
        raise LipCacheError(status, msg.decode() if msg else "")
