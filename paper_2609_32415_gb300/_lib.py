"""ctypes view of librefadapt.so: structures and prototypes of include/refadapt.h.

The library is built in-tree by ``paper_2609_32415_gb300.build``. Loading fails
loudly when it is missing: there is no CPU fallback for any entry point.
"""
import ctypes
import os
from ctypes import POINTER, c_double, c_float, c_int32, c_int64, c_size_t, c_uint64, c_void_p

PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(PKG, "librefadapt.so")

RA_OK, RA_EINVAL, RA_EUNSUPPORTED, RA_ECUDA, RA_ETIMEOUT = 0, 1, 2, 3, 4
RA_MODE_REUSE, RA_MODE_BOUNDARY, RA_MODE_COMPUTE, RA_MODE_FULL = 0, 1, 2, 3
RA_TEXT, RA_REF, RA_TGT = 0, 1, 2
RA_CUE_PRODUCT, RA_CUE_CHANGE, RA_CUE_EXPOSURE = 0, 1, 2
RA_MASS_TILE_ROWS = 128
RA_Q_DELTA_NOALLOC_MAX_BH = 96

EXPORTED = (
    "refadapt_joint_attn", "refadapt_mass_partial_len", "refadapt_q_delta_workspace_size",
    "refadapt_q_delta", "refadapt_state_size", "refadapt_state_init", "refadapt_gate",
    "refadapt_ref_cache_update", "refadapt_status_string", "refadapt_last_error",
    "refadapt_set_wait_budget_ns", "refadapt_check_error", "refadapt_version",
    "refadapt_selftest_wait_timeout", "refadapt_q_delta_noalloc", "refadapt_rope_table",
    "refadapt_ln_modulate", "refadapt_gemm", "refadapt_q_delta_gate",
)
RA_EPI_STORE, RA_EPI_GELU, RA_EPI_RESID, RA_EPI_QKV = 0, 1, 2, 3


class RaSeg(ctypes.Structure):
    _fields_ = [("ptr", c_void_p), ("stride_b", c_int64), ("stride_h", c_int64),
                ("stride_n", c_int64), ("n", c_int32), ("reserved", c_int32)]


class RaAttnArgs(ctypes.Structure):
    _fields_ = [("B", c_int32), ("H", c_int32), ("d", c_int32), ("mass_rows", c_int32),
                ("q", RaSeg * 3), ("k", RaSeg * 3), ("v", RaSeg * 3), ("o", RaSeg * 3),
                ("softmax_scale", c_float), ("mass_row_stride", c_int32),
                ("ref_logit_bias", c_void_p), ("mode", c_void_p), ("mass_partial", c_void_p),
                ("err_word", c_void_p), ("ref_fresh_q", RaSeg), ("ref_fresh_k", RaSeg), ("ref_fresh_v", RaSeg),
                ("a_b", c_void_p), ("step", c_int32), ("reserved", c_int32)]


class RaGateArgs(ctypes.Structure):
    _fields_ = [("theta", c_double), ("t", c_int32), ("b", c_int32), ("B", c_int32), ("H", c_int32),
                ("delta_max", c_int32), ("forced_boundary", c_int32), ("mass_partial_len", c_int32),
                ("mass_row_count", c_int32), ("cue", c_int32), ("reserved", c_int32),
                ("q_delta", c_void_p), ("mass_partial_prev", c_void_p),
                ("state", c_void_p), ("mode_out", c_void_p), ("gbar_out", c_void_p),
                ("m_out", c_void_p)]


class RaLnmodSeg(ctypes.Structure):
    _fields_ = [("h", c_void_p), ("h_stride_s", c_int64), ("h_stride_r", c_int64),
                ("x", c_void_p), ("x_stride_s", c_int64), ("x_stride_r", c_int64),
                ("shift", c_void_p), ("scale", c_void_p), ("mod_stride_s", c_int64),
                ("rows", c_int32), ("gated", c_int32)]


class RaLnmodArgs(ctypes.Structure):
    _fields_ = [("B", c_int32), ("C", c_int32), ("n_seg", c_int32), ("reserved", c_int32),
                ("eps", c_float), ("reserved2", c_float), ("seg", RaLnmodSeg * 3), ("mode", c_void_p)]


class RaGemmSeg(ctypes.Structure):
    _fields_ = [("a", c_void_p), ("a_stride_s", c_int64), ("a_stride_r", c_int64),
                ("rows", c_int32), ("gated", c_int32), ("w", c_void_p), ("bias", c_void_p),
                ("out", c_void_p), ("out_stride_s", c_int64), ("out_stride_r", c_int64),
                ("resid", c_void_p), ("resid_stride_s", c_int64), ("resid_stride_r", c_int64),
                ("gate", c_void_p), ("gate_stride_s", c_int64),
                ("q_out", RaSeg), ("k_out", RaSeg), ("v_out", RaSeg),
                ("q_norm", c_void_p), ("k_norm", c_void_p), ("pos_offset", c_int32), ("reserved", c_int32)]


class RaGemmArgs(ctypes.Structure):
    _fields_ = [("B", c_int32), ("N", c_int32), ("K", c_int32), ("epilogue", c_int32),
                ("H", c_int32), ("d", c_int32), ("n_seg", c_int32), ("rope_len", c_int32),
                ("seg", RaGemmSeg * 3), ("mode", c_void_p), ("rope", c_void_p),
                ("norm_eps", c_float), ("tile_mode", c_int32), ("err_word", c_void_p)]


class RefAdaptError(RuntimeError):
    def __init__(self, fn, status, msg):
        super().__init__("%s failed: %s (%s)" % (fn, _status_name(status), msg))
        self.status = status


def _status_name(s):
    return {0: "RA_OK", 1: "RA_EINVAL", 2: "RA_EUNSUPPORTED", 3: "RA_ECUDA", 4: "RA_ETIMEOUT"}.get(s, str(s))


_lib = None


def load():
    """Load librefadapt.so (raises if it has not been built)."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(LIB_PATH):
        raise RuntimeError(
            "librefadapt.so is missing (%s): build it with `python -c \"import __graft_entry__ as g; "
            "g.build()\"` or `python -m paper_2609_32415_gb300.build`; there is no CPU fallback" % LIB_PATH)
    lib = ctypes.CDLL(LIB_PATH)
    lib.refadapt_joint_attn.restype = c_int32
    lib.refadapt_joint_attn.argtypes = [POINTER(RaAttnArgs), c_void_p]
    lib.refadapt_mass_partial_len.restype = c_int32
    lib.refadapt_mass_partial_len.argtypes = [c_int32, c_int32]
    lib.refadapt_q_delta_workspace_size.restype = c_size_t
    lib.refadapt_q_delta_workspace_size.argtypes = [c_int32, c_int32]
    lib.refadapt_q_delta.restype = c_int32
    lib.refadapt_q_delta.argtypes = [POINTER(RaSeg), POINTER(RaSeg), c_int32, c_int32, c_int32, c_float,
                                     c_void_p, c_void_p, c_size_t, c_void_p]
    lib.refadapt_state_size.restype = c_size_t
    lib.refadapt_state_size.argtypes = [c_int32]
    lib.refadapt_state_init.restype = c_int32
    lib.refadapt_state_init.argtypes = [c_void_p, c_int32, c_void_p]
    lib.refadapt_gate.restype = c_int32
    lib.refadapt_gate.argtypes = [POINTER(RaGateArgs), c_void_p]
    lib.refadapt_q_delta_gate.restype = c_int32
    lib.refadapt_q_delta_gate.argtypes = [POINTER(RaSeg), POINTER(RaSeg), c_int32, c_int32, c_int32, c_float,
                                          c_void_p, c_void_p, c_size_t, POINTER(RaGateArgs), c_void_p]
    lib.refadapt_ref_cache_update.restype = c_int32
    lib.refadapt_ref_cache_update.argtypes = [POINTER(RaSeg), POINTER(RaSeg), POINTER(RaSeg), POINTER(RaSeg),
                                              c_int32, c_int32, c_int32, POINTER(RaSeg), POINTER(RaSeg),
                                              c_int32, c_int32, c_void_p, c_int32, c_void_p, c_void_p]
    lib.refadapt_status_string.restype = ctypes.c_char_p
    lib.refadapt_status_string.argtypes = [c_int32]
    lib.refadapt_last_error.restype = ctypes.c_char_p
    lib.refadapt_last_error.argtypes = []
    lib.refadapt_set_wait_budget_ns.restype = None
    lib.refadapt_set_wait_budget_ns.argtypes = [c_uint64]
    lib.refadapt_check_error.restype = c_int32
    lib.refadapt_check_error.argtypes = [c_void_p, c_void_p]
    lib.refadapt_version.restype = c_int32
    lib.refadapt_version.argtypes = []
    lib.refadapt_q_delta_noalloc.restype = c_int32
    lib.refadapt_q_delta_noalloc.argtypes = [POINTER(RaSeg), POINTER(RaSeg), c_int32, c_int32, c_int32, c_float,
                                             c_void_p, c_void_p]
    lib.refadapt_rope_table.restype = c_int32
    lib.refadapt_rope_table.argtypes = [c_void_p, c_int32, c_int32, c_double, c_void_p]
    lib.refadapt_ln_modulate.restype = c_int32
    lib.refadapt_ln_modulate.argtypes = [POINTER(RaLnmodArgs), c_void_p]
    lib.refadapt_gemm.restype = c_int32
    lib.refadapt_gemm.argtypes = [POINTER(RaGemmArgs), c_void_p]
    lib.refadapt_selftest_wait_timeout.restype = c_int32
    lib.refadapt_selftest_wait_timeout.argtypes = [c_void_p, c_uint64, c_void_p]
    _lib = lib
    return lib


def check(fn, status):
    if status != RA_OK:
        msg = load().refadapt_last_error().decode(errors="replace")
        raise RefAdaptError(fn, status, msg)
    return status
