"""ctypes view of the AGN C ABI (include/agn.h): library loading and signatures.

The library is built in-tree (`_build/libagn_gb300.so`, see build.py).  There
is no fallback: if it is missing, loading raises.  With AGN_LIB_VARIANT=check
in the environment the bounds-checked build (`_build_check/
libagn_gb300_check.so`) is loaded instead.
"""

from __future__ import annotations

import ctypes as C
import os

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "_build", "libagn_gb300.so")
LIB_CHECK_PATH = os.path.join(HERE, "_build_check", "libagn_gb300_check.so")

AGN_OK = 0
AGN_E_INVALID = -1
AGN_E_SCHEDULE = -2
AGN_E_OOM = -3
AGN_E_CUDA = -4
AGN_E_TIMEOUT = -5
AGN_E_NONFINITE = -6
AGN_E_UNSUPPORTED = -7
AGN_E_BOUNDS = -8

AGN_PREC_FP32 = 0
AGN_PREC_BF16 = 1
AGN_DIST_UNIFORM = 0
AGN_DIST_NORMAL = 1
AGN_OPT_SGD = 0
AGN_OPT_ADAM = 1
AGN_COMMIT_AGN = 0
AGN_COMMIT_DYNSGD = 1
AGN_GEMM_AUTO = 0
AGN_GEMM_SIMT = 1
AGN_GEMM_TCGEN05 = 2

KERNEL_CLASSES = ["gather", "forward", "softmax", "backward_dx", "backward_dw", "commit",
                  "norms", "other", "forward_head"]

ERROR_NAMES = {
    AGN_E_INVALID: "AGN_E_INVALID", AGN_E_SCHEDULE: "AGN_E_SCHEDULE", AGN_E_OOM: "AGN_E_OOM",
    AGN_E_CUDA: "AGN_E_CUDA", AGN_E_TIMEOUT: "AGN_E_TIMEOUT",
    AGN_E_NONFINITE: "AGN_E_NONFINITE", AGN_E_UNSUPPORTED: "AGN_E_UNSUPPORTED",
    AGN_E_BOUNDS: "AGN_E_BOUNDS",
}


class agn_options(C.Structure):
    _fields_ = [
        ("precision", C.c_int32),
        ("batch", C.c_int32),
        ("n_samples", C.c_int64),
        ("input_dist", C.c_int32),
        ("teacher_dims", C.POINTER(C.c_int32)),
        ("n_teacher_dims", C.c_int32),
        ("normalize", C.c_int32),
        ("gemm", C.c_int32),
        ("tau_lo", C.c_int32),
        ("tau_hi", C.c_int32),
        ("stream", C.c_void_p),
        ("x_init", C.POINTER(C.c_float)),
        ("y_init", C.POINTER(C.c_int32)),
        ("theta_init", C.POINTER(C.c_float)),
        ("tc_mask", C.c_int32),
        ("commit_rule", C.c_int32),
        ("elide_accumulator", C.c_int32),
        ("n_eval", C.c_int64),
        ("local_optimizer", C.c_int32),
        ("adam_beta1", C.c_float),
        ("adam_beta2", C.c_float),
        ("adam_eps", C.c_float),
    ]


_I32P = C.POINTER(C.c_int32)
_I64P = C.POINTER(C.c_int64)
_F32P = C.POINTER(C.c_float)
_F64P = C.POINTER(C.c_double)

# name -> (restype, argtypes); every symbol the header declares.
SIGNATURES = {
    "agn_default_options": (None, [C.POINTER(agn_options)]),
    "agn_create": (C.c_int, [_I32P, C.c_int32, C.c_int32, C.c_int32, C.c_double, C.c_uint64,
                             C.POINTER(agn_options), C.POINTER(C.c_void_p)]),
    "agn_run": (C.c_int, [C.c_void_p, C.c_int32, _I32P, _I32P, C.c_int32]),
    "agn_central": (C.c_int, [C.c_void_p, _F32P, C.c_int64]),
    "agn_replica": (C.c_int, [C.c_void_p, C.c_int32, _F32P, C.c_int64]),
    "agn_loss": (C.c_int, [C.c_void_p, _F32P, C.c_int64]),
    "agn_delta_norm": (C.c_int, [C.c_void_p, _F32P, C.c_int64]),
    "agn_evaluate": (C.c_int, [C.c_void_p, _F32P, _F32P, _I32P, C.c_int64]),
    "agn_temporal_efficiency": (C.c_int, [_F64P, _F64P, C.c_int64, _F64P, _F64P, C.c_int64,
                                          _F64P]),
    "agn_num_params": (C.c_int64, [C.c_void_p]),
    "agn_num_commits": (C.c_int64, [C.c_void_p]),
    "agn_last_run_stats": (C.c_int, [C.c_void_p, _F64P, C.c_int64]),
    "agn_generate_inputs": (C.c_int, [_I32P, C.c_int32, C.c_int32, _I32P, C.c_int32, C.c_uint64,
                                      C.c_int64, C.c_int64, _F32P, _I32P, _F32P]),
    "agn_export_inputs": (C.c_int, [C.c_void_p, _F32P, _I32P, _F32P]),
    "agn_profile": (C.c_int, [C.c_void_p, C.c_int32]),
    "agn_kernel_stats": (C.c_int, [C.c_void_p, _F64P, C.c_int64]),
    "agn_last_error": (C.c_char_p, [C.c_void_p]),
    "agn_destroy": (None, [C.c_void_p]),
    "agn_make_schedule": (C.c_int, [C.c_int32, C.c_int32, C.c_int32, C.c_int32, C.c_uint64,
                                    _I32P, _I32P]),
    "agn_plan_waves": (C.c_int, [C.c_int32, C.c_int32, C.c_int32, _I32P, _I32P, C.c_int32,
                                 _I32P, _I32P, _I32P, _I32P, _I64P, C.c_int64, _I32P, _I32P,
                                 _I64P]),
    "agn_commit_pull": (C.c_int, [C.c_void_p, C.c_void_p, C.c_void_p, C.c_void_p, C.c_int64,
                                  C.c_int64, C.c_int32, C.c_int32, _I32P, _I32P, _I32P,
                                  C.c_double, C.c_int32, C.c_int32, C.c_void_p, C.c_void_p]),
    "agn_commit_pull_noalloc": (C.c_int, [C.c_void_p, C.c_void_p, C.c_void_p, C.c_void_p,
                                          C.c_int64, C.c_int64, C.c_int32, C.c_int32, _I32P,
                                          _I32P, _I32P, C.c_double, C.c_int32, C.c_int32,
                                          C.c_void_p, C.c_void_p]),
    "agn_debug_waits": (C.c_int, [C.c_void_p, C.c_int64, C.c_int32]),
    "agn_fill_commit_inputs": (C.c_int, [C.c_void_p, C.c_void_p, C.c_void_p, C.c_int64,
                                         C.c_int64, C.c_int32, C.c_uint64, C.c_void_p]),
}

_LIB = None


def library_file() -> str:
    """The library this process loads: the bounds-checked build when
    AGN_LIB_VARIANT=check, else the normal one."""
    return LIB_CHECK_PATH if os.environ.get("AGN_LIB_VARIANT") == "check" else LIB_PATH


def load():
    """Load the library (once) and declare every signature; raise if missing."""
    global _LIB
    if _LIB is None:
        path = library_file()
        if not os.path.exists(path):
            raise RuntimeError(
                f"AGN CUDA library not found at {path}; build it first "
                "(python -c 'import __graft_entry__ as g; g.build()')")
        lib = C.CDLL(path)
        for name, (res, args) in SIGNATURES.items():
            fn = getattr(lib, name)
            fn.restype = res
            fn.argtypes = args
        _LIB = lib
    return _LIB
