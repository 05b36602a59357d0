"""ctypes declarations mirroring include/rdn.h (structs and entry points)."""
from __future__ import annotations

import ctypes
import os

from . import build as _build

P = ctypes.c_void_p
F = ctypes.POINTER(ctypes.c_float)

RDN_F32, RDN_BF16 = 0, 1
RDN_FLAG_SAVE_FOR_BWD = 0x1  # rdn_fwd_args.flags (include/rdn.h)
RDN_FLAG_TIED_GAMMA = 0x2
# the paper's variants of the method
RDN_FLAG_DECAYED_RESIDUAL = 0x4
RDN_FLAG_PLAIN_COMBINE = 0x8
RDN_FLAG_TANH_RESIDUAL = 0x10
RDN_FLAG_STATELESS_AUX = 0x20
RDN_FLAG_VARIANTS = 0x3C
RDN_FLAG_F32_OUT = 0x40  # fp32 results for bf16 inputs
RDN_FLAG_QK_NORM = 0x80  # q, k are raw x: SiLU + L2 normalisation applied in the library

STATUS = {0: "RDN_OK", 1: "RDN_ERR_INVALID_ARG", 2: "RDN_ERR_UNSUPPORTED", 3: "RDN_ERR_CUDA",
          4: "RDN_ERR_TIMEOUT", 5: "RDN_ERR_WORKSPACE", 6: "RDN_ERR_MISALIGNED"}

# every function the header declares (checked by the CPU tests)
EXPORTS = ["rla_fwd", "rdn_fwd", "rla_bwd", "rdn_bwd", "rdn_decode_step", "rla_fwd_workspace_size",
           "rdn_fwd_workspace_size", "rla_bwd_workspace_size", "rdn_bwd_workspace_size",
           "rdn_last_error", "rdn_version", "rdn_prof_start", "rdn_prof_stop", "rdn_fwd_noalloc",
           "rdn_qk_prologue", "rdn_qk_prologue_bwd", "rdn_chunk_slots", "rdn_device_status"]


class ProfRecord(ctypes.Structure):
    _fields_ = [("name", ctypes.c_char * 40), ("ms", ctypes.c_float)]


class FwdArgs(ctypes.Structure):
    _fields_ = [("B", ctypes.c_int), ("T", ctypes.c_int), ("H", ctypes.c_int),
                ("Dk", ctypes.c_int), ("Dv", ctypes.c_int), ("dtype", ctypes.c_int),
                ("q", P), ("k", P), ("v", P), ("g", P), ("beta", P), ("gamma", P),
                ("clip", ctypes.c_float), ("S0", P), ("R0", P), ("o", P),
                ("ST", P), ("RT", P), ("S_chunks", P), ("R_chunks", P),
                ("scale", ctypes.c_float), ("flags", ctypes.c_uint),
                ("workspace", P), ("workspace_bytes", ctypes.c_size_t),
                ("cu_seqlens", P), ("num_seqs", ctypes.c_int), ("qk_eps", ctypes.c_float)]


class BwdArgs(ctypes.Structure):
    _fields_ = [("fwd", FwdArgs), ("dO", P), ("dST", P), ("dRT", P),
                ("dq", P), ("dk", P), ("dv", P), ("dg", P), ("dbeta", P), ("dgamma", P),
                ("dS0", P), ("dR0", P), ("workspace", P), ("workspace_bytes", ctypes.c_size_t)]


class DecodeArgs(ctypes.Structure):
    _fields_ = [("N", ctypes.c_int), ("H", ctypes.c_int), ("Dk", ctypes.c_int),
                ("Dv", ctypes.c_int), ("dtype", ctypes.c_int), ("variant", ctypes.c_int),
                ("q", P), ("k", P), ("v", P), ("g", P), ("beta", P), ("gamma", P),
                ("clip", ctypes.c_float), ("scale", ctypes.c_float),
                ("S", P), ("R", P), ("o", P), ("flags", ctypes.c_uint),
                ("qk_eps", ctypes.c_float)]


class PrologueArgs(ctypes.Structure):
    _fields_ = [("rows", ctypes.c_longlong), ("D", ctypes.c_int), ("dtype", ctypes.c_int),
                ("eps", ctypes.c_float), ("x", P * 2), ("y", P * 2), ("dy", P * 2),
                ("dx", P * 2)]


_lib = None


def lib_path() -> str:
    return _build.LIB


def load(build_if_missing: bool = True):
    """Load librdn.so (building it first if needed and allowed)."""
    global _lib
    if _lib is not None:
        return _lib
    path = _build.LIB
    if not os.path.exists(path) or (build_if_missing and not _build.up_to_date()):
        if not build_if_missing:
            raise RuntimeError(f"librdn.so not built ({path}); run paper_2509_25223_gb300.build")
        _build.build()
    lib = ctypes.CDLL(path)
    S = ctypes.c_int
    for name, argt in [("rla_fwd", [ctypes.POINTER(FwdArgs), P]),
                       ("rdn_fwd", [ctypes.POINTER(FwdArgs), P]),
                       ("rdn_fwd_noalloc", [ctypes.POINTER(FwdArgs), P]),
                       ("rla_bwd", [ctypes.POINTER(BwdArgs), P]),
                       ("rdn_bwd", [ctypes.POINTER(BwdArgs), P]),
                       ("rdn_decode_step", [ctypes.POINTER(DecodeArgs), P]),
                       ("rdn_qk_prologue", [ctypes.POINTER(PrologueArgs), P]),
                       ("rdn_qk_prologue_bwd", [ctypes.POINTER(PrologueArgs), P]),
                       ("rla_fwd_workspace_size", [ctypes.POINTER(FwdArgs), ctypes.POINTER(ctypes.c_size_t)]),
                       ("rdn_fwd_workspace_size", [ctypes.POINTER(FwdArgs), ctypes.POINTER(ctypes.c_size_t)]),
                       ("rla_bwd_workspace_size", [ctypes.POINTER(BwdArgs), ctypes.POINTER(ctypes.c_size_t)]),
                       ("rdn_bwd_workspace_size", [ctypes.POINTER(BwdArgs), ctypes.POINTER(ctypes.c_size_t)]),
                       ("rdn_chunk_slots", [ctypes.POINTER(FwdArgs), ctypes.POINTER(ctypes.c_longlong)])]:
        fn = getattr(lib, name)
        fn.argtypes = argt
        fn.restype = S
    lib.rdn_prof_start.argtypes = [ctypes.c_int]
    lib.rdn_prof_start.restype = S
    lib.rdn_prof_stop.argtypes = [ctypes.POINTER(ProfRecord), ctypes.c_int,
                                  ctypes.POINTER(ctypes.c_int)]
    lib.rdn_prof_stop.restype = S
    lib.rdn_device_status.argtypes = [P, ctypes.POINTER(ctypes.c_int)]
    lib.rdn_device_status.restype = S
    lib.rdn_last_error.restype = ctypes.c_char_p
    lib.rdn_last_error.argtypes = []
    lib.rdn_version.restype = ctypes.c_char_p
    lib.rdn_version.argtypes = []
    _lib = lib
    return lib
