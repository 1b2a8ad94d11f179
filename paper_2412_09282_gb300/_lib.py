"""ctypes declarations of the C ABI in include/crvq.h (libcrvq.so, built in-tree)."""
from __future__ import annotations

import ctypes as C
import os

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "libcrvq.so")

c_f32p = C.POINTER(C.c_float)
c_i32p = C.POINTER(C.c_int32)
c_i64p = C.POINTER(C.c_int64)
c_f64p = C.POINTER(C.c_double)
c_vp = C.c_void_p


class crvq_codebook(C.Structure):
    _fields_ = [("C", c_vp), ("K", C.c_int32), ("_pad", C.c_int32), ("codes", c_vp),
                ("ld", C.c_int64), ("G_cov", C.c_int64)]


class crvq_config(C.Structure):
    _fields_ = [("d", C.c_int32), ("K_base", C.c_int32), ("n_ext", C.c_int32),
                ("K_ext", C.c_int32), ("crit_frac", C.c_float), ("B", C.c_int32),
                ("kmeans_iters", C.c_int32), ("refine_rounds", C.c_int32),
                ("eps_rel", C.c_float), ("damp_rel", C.c_float),
                ("importance_mode", C.c_int32), ("n_base", C.c_int32), ("seed", C.c_uint64)]


class crvq_layer_outputs(C.Structure):
    _fields_ = [("perm", c_vp), ("C_base", c_vp), ("codes_base", c_vp), ("C_ext", c_vp),
                ("codes_ext", c_vp), ("W_hat", c_vp), ("importance", c_vp)]


class crvq_layer_report(C.Structure):
    _fields_ = [("loss_pre", C.c_double), ("loss_block", C.c_double),
                ("loss_crit", C.c_double), ("loss_full", C.c_double),
                ("loss_before_refine", C.c_double), ("scores", C.c_double),
                ("n_crit_groups", C.c_int64), ("flagged", C.c_int64),
                ("refine_rounds_done", C.c_int32),
                ("_pad", C.c_int32)]


class crvq_kernel_stat(C.Structure):
    _fields_ = [("name", C.c_char * 64), ("launches", C.c_int64), ("ms", C.c_double),
                ("units", C.c_double)]


# name -> (restype, argtypes)
SIGNATURES = {
    "crvq_last_error": (C.c_char_p, []),
    "crvq_version": (C.c_char_p, []),
    "crvq_sync": (C.c_int32, [c_vp]),
    "crvq_profile_begin": (C.c_int32, []),
    "crvq_profile_end": (C.c_int32, [C.POINTER(crvq_kernel_stat), C.c_int32, c_i32p]),
    "crvq_profile_filter": (C.c_int32, [C.c_char_p]),
    "crvq_launch_count": (C.c_int64, []),
    "crvq_selftest_bounded_wait": (C.c_int32, [c_vp]),
    "crvq_hessian": (C.c_int32, [c_vp, C.c_int64, C.c_int64, C.c_int32, C.c_float, c_vp, c_vp,
                                 c_vp, c_vp, c_vp]),
    "crvq_hessian_blocks": (C.c_int32, [c_vp, C.c_int64, C.c_int64, C.c_int32, C.c_float,
                                        c_vp, c_vp, c_vp, c_vp, c_vp]),
    "crvq_hessian_inverse_diag": (C.c_int32, [c_vp, C.c_int64, c_vp, c_vp]),
    "crvq_select_reorder_channels": (C.c_int32, [c_vp, C.c_int64, C.c_int64, C.c_int32, c_vp,
                                                 c_vp, c_vp, C.c_float, C.c_int32, C.c_uint64,
                                                 c_vp, c_vp, c_vp, c_vp, c_i64p, c_vp]),
    "crvq_kmeans_init": (C.c_int32, [c_vp, C.c_int64, C.c_int64, C.c_int64, C.c_int32,
                                     C.POINTER(crvq_codebook), C.c_int32, C.c_int32,
                                     C.c_uint64, c_vp, c_vp]),
    "crvq_encode_beam": (C.c_int32, [c_vp, C.c_int64, C.c_int64, C.c_int64, C.c_int32, c_vp,
                                     C.POINTER(crvq_codebook), C.c_int32, C.c_int32, C.c_int32,
                                     C.c_int32, c_vp, c_vp]),
    "crvq_update_codebook": (C.c_int32, [c_vp, C.c_int64, C.c_int64, C.c_int64, C.c_int32,
                                         c_vp, C.POINTER(crvq_codebook), C.c_int32, C.c_int32,
                                         c_vp, c_vp, c_vp]),
    "crvq_update_codebook_noalloc": (C.c_int32, [c_vp, C.c_int64, C.c_int64, C.c_int64,
                                                 C.c_int32, c_vp, C.POINTER(crvq_codebook),
                                                 C.c_int32, C.c_int32, c_vp, c_vp, c_vp]),
    "crvq_reconstruct_error": (C.c_int32, [c_vp, C.c_int64, C.c_int64, C.c_int32, c_vp, c_vp,
                                           C.POINTER(crvq_codebook), C.c_int32, C.c_int64,
                                           c_vp, C.c_int64, C.c_double, c_vp, c_f64p, c_vp]),
    "crvq_coupled_sweep": (C.c_int32, [c_vp, C.c_int64, C.c_int64, C.c_int32, c_vp,
                                       C.POINTER(crvq_codebook), C.c_int32, C.c_int32,
                                       C.c_int32, c_f64p, c_vp]),
    "crvq_lut_matvec": (C.c_int32, [c_vp, C.c_int64, C.c_int64, C.c_int64, C.c_int32, c_vp,
                                    C.POINTER(crvq_codebook), C.c_int32, C.c_int64, c_vp,
                                    C.c_int64, c_vp]),
    "crvq_avg_bits": (C.c_double, [C.c_int32, C.c_int32, C.c_int32, C.c_double, C.c_int64,
                                   C.c_int64, C.c_int32]),
    "crvq_avg_bits_bases": (C.c_double, [C.c_int32, C.c_int32, C.c_int32, C.c_int32,
                                         C.c_double, C.c_int64, C.c_int64, C.c_int32]),
    "crvq_n_crit_groups": (C.c_int64, [C.c_int64, C.c_int32, C.c_float]),
    "crvq_quantize_layer": (C.c_int32, [c_vp, c_vp, C.c_int64, C.c_int64, C.c_int64,
                                        C.POINTER(crvq_config), C.POINTER(crvq_layer_outputs),
                                        C.POINTER(crvq_layer_report), c_vp]),
}

_lib = None


def load():
    """Loads libcrvq.so (raises if it has not been built: there is no fallback)."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise ImportError(
                f"{LIB_PATH} is missing: build it with `python -m paper_2412_09282_gb300.build` "
                "(nvcc, sm_103a). The CRVQ kernels have no CPU fallback.")
        lib = C.CDLL(LIB_PATH)
        for name, (res, args) in SIGNATURES.items():
            fn = getattr(lib, name)
            fn.restype = res
            fn.argtypes = args
        _lib = lib
    return _lib
