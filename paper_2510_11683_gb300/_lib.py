"""ctypes declarations of the C ABI in include/bgpo.h (argument marshalling only)."""
import ctypes
import os

from .build import CHECKED_LIB_PATH, LIB_PATH

c_int32 = ctypes.c_int32
c_void_p = ctypes.c_void_p
c_size_t = ctypes.c_size_t

BGPO_OK = 0
STATUS_NAMES = {
    0: "BGPO_OK", 1: "BGPO_ERR_INVALID_ARG", 2: "BGPO_ERR_SHAPE", 3: "BGPO_ERR_ALIGNMENT",
    4: "BGPO_ERR_WORKSPACE_TOO_SMALL", 5: "BGPO_ERR_NONFINITE", 6: "BGPO_ERR_UNSUPPORTED_DEVICE",
    7: "BGPO_ERR_CUDA", 8: "BGPO_ERR_TIMEOUT", 9: "BGPO_ERR_BOUNDS",
}


class BgpoProblem(ctypes.Structure):
    """Mirror of ``struct bgpo_problem``."""
    _fields_ = [
        ("B", c_int32), ("P", c_int32), ("R", c_int32), ("H", c_int32), ("V", c_int32),
        ("n_t", c_int32), ("G", c_int32), ("t_mode", c_int32),
        ("seed", ctypes.c_uint64), ("loss_scale", ctypes.c_float), ("b_offset", c_int32),
        ("trace", c_void_p), ("resp_len", c_void_p),
        ("flags", ctypes.c_uint32), ("vocab_chunk", c_int32),
    ]


# name -> (restype, argtypes); every symbol include/bgpo.h declares
SIGNATURES = {
    "bgpo_abi_version": (c_int32, []),
    "bgpo_status_string": (ctypes.c_char_p, [c_int32]),
    "bgpo_validate_problem": (c_int32, [ctypes.POINTER(BgpoProblem)]),
    "bgpo_workspace_bytes": (c_size_t, [ctypes.POINTER(BgpoProblem)]),
    "bgpo_sample_mask": (c_int32, [ctypes.POINTER(BgpoProblem), c_int32, c_void_p, c_size_t,
                                   c_void_p, c_void_p, c_void_p]),
    "bgpo_elbo_fwd": (c_int32, [ctypes.POINTER(BgpoProblem), c_int32, c_void_p, c_void_p, c_void_p,
                                c_void_p, c_size_t, c_void_p, c_void_p]),
    "bgpo_bound_coeffs": (c_int32, [ctypes.POINTER(BgpoProblem), c_int32, c_void_p, c_void_p,
                                    c_void_p, c_void_p, c_void_p, c_void_p, c_size_t, c_void_p]),
    "bgpo_vrpo_coeffs": (c_int32, [ctypes.POINTER(BgpoProblem), c_void_p, c_void_p, c_void_p,
                                   c_void_p, c_void_p, c_void_p, c_size_t, c_void_p]),
    "bgpo_elbo_bwd_accumulate": (c_int32, [ctypes.POINTER(BgpoProblem), c_int32, c_void_p, c_void_p,
                                           c_void_p, c_void_p, c_void_p, c_size_t, c_void_p,
                                           c_void_p, c_void_p]),
    "bgpo_group_advantage": (c_int32, [ctypes.POINTER(BgpoProblem), c_void_p, c_void_p, c_void_p]),
    "bgpo_elbo_fwd_noalloc": (c_int32, [ctypes.POINTER(BgpoProblem), c_int32, c_void_p, c_void_p,
                                        c_void_p, c_void_p, c_void_p, c_void_p]),
    "bgpo_get_device_error": (c_int32, [c_void_p, c_size_t, ctypes.POINTER(c_int32),
                                        ctypes.POINTER(c_int32), c_void_p]),
    "bgpo_clear_device_error": (c_int32, [c_void_p, c_size_t, c_void_p]),
    "bgpo_selftest_bounded_wait": (c_int32, [c_void_p, c_size_t, ctypes.c_uint32, c_void_p]),
    "bgpo_trace_create": (c_void_p, [c_int32]),
    "bgpo_trace_destroy": (None, [c_void_p]),
    "bgpo_trace_reset": (None, [c_void_p]),
    "bgpo_trace_count": (c_int32, [c_void_p]),
    "bgpo_trace_get": (c_int32, [c_void_p, c_int32, ctypes.POINTER(c_int32),
                                 ctypes.POINTER(ctypes.c_float)]),
    "bgpo_kernel_name": (ctypes.c_char_p, [c_int32]),
}

_LIB = None


class BgpoError(RuntimeError):
    def __init__(self, fn, status):
        self.status = status
        super().__init__(f"{fn} failed: {STATUS_NAMES.get(status, status)}")


def lib_path():
    """lib/libbgpo.so, or with BGPO_LIBRARY=checked in the environment the
    bounds-checked build lib/libbgpo_checked.so."""
    choice = os.environ.get("BGPO_LIBRARY", "")
    if choice not in ("", "checked"):
        raise ValueError(f"BGPO_LIBRARY must be unset or 'checked', got {choice!r}")
    return CHECKED_LIB_PATH if choice == "checked" else LIB_PATH


def lib():
    """Loads the library lib_path() names (built by build.py); raises if it is missing."""
    global _LIB
    if _LIB is None:
        path = lib_path()
        if not os.path.exists(path):
            raise ImportError(
                f"CUDA library {path} is missing: build it with "
                "`python -c 'import __graft_entry__ as g; g.build()'` "
                "or `python -m paper_2510_11683_gb300.build [--checked]`")
        h = ctypes.CDLL(path)
        for name, (res, args) in SIGNATURES.items():
            f = getattr(h, name)
            f.restype = res
            f.argtypes = args
        _LIB = h
    return _LIB


def check(fn, status):
    if status != BGPO_OK:
        raise BgpoError(fn, status)
