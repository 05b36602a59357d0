"""GB300 (sm_103a) layer hot path of Residual Linear Attention (RLA) and
Residual Delta Net (RDN), arXiv 2509.25223, Section 3.4.

A thin binding over the C ABI in include/rdn.h (librdn.so): it marshals torch
tensor pointers, sizes and the current CUDA stream, allocates the workspace
the library asks for, and raises on a non-OK status.  Every step of the
computation runs in the library's CUDA kernels; there is no CPU or PyTorch
fallback, and a missing or unloadable library is an error.

Tensors (contiguous, on one CUDA device):
    q, k [B,T,H,Dk]; v [B,T,H,Dv]            bf16 or fp32 (same dtype)
    g (log-decay = log alpha), beta, gamma [B,T,H]   fp32
    S0, R0 [B,H,Dk,Dv] fp32 or None
Results: o [B,T,H,Dv] in the input dtype; ST, RT [B,H,Dk,Dv] fp32.
"""
from __future__ import annotations

import ctypes
import math

import torch

from . import _abi
from ._abi import BwdArgs, DecodeArgs, FwdArgs
# variant flags (variant_flags= of the forward and backward calls): residual
# against a_t S_{t-1} k_t; ungated combine S_{t-1} q + R_t q; c tanh(x / c)
# residual; stateless correction R_t = r_t k_t^T
from ._abi import (RDN_FLAG_DECAYED_RESIDUAL as DECAYED_RESIDUAL,  # noqa: F401
                   RDN_FLAG_PLAIN_COMBINE as PLAIN_COMBINE,
                   RDN_FLAG_STATELESS_AUX as STATELESS_AUX,
                   RDN_FLAG_TANH_RESIDUAL as TANH_RESIDUAL)

__all__ = ["rla_fwd", "rdn_fwd", "rla_bwd", "rdn_bwd", "qk_prologue", "qk_prologue_bwd", "rdn_decode_step", "RdnError", "library",
           "CHUNK"]

CHUNK = 64


class RdnError(RuntimeError):
    def __init__(self, fn, status, msg):
        super().__init__(f"{fn} -> {_abi.STATUS.get(status, status)}: {msg}")
        self.status = status


def library():
    """The loaded librdn.so (ctypes.CDLL)."""
    return _abi.load()


def _check(fn, st):
    if st != 0:
        raise RdnError(fn, st, _abi.load().rdn_last_error().decode())


def _ptr(t):
    if t is None:
        return None
    if not t.is_cuda:
        raise ValueError("rdn: tensors must be on a CUDA device")
    if not t.is_contiguous():
        raise ValueError("rdn: tensors must be contiguous")
    return ctypes.c_void_p(t.data_ptr())


def _dtype_code(t):
    if t.dtype == torch.bfloat16:
        return _abi.RDN_BF16
    if t.dtype == torch.float32:
        return _abi.RDN_F32
    raise ValueError(f"rdn: unsupported dtype {t.dtype}")


def _stream(t):
    return ctypes.c_void_p(torch.cuda.current_stream(t.device).cuda_stream)


def _alloc_ws(nbytes, device):
    if nbytes == 0:
        return None
    return torch.empty(nbytes, dtype=torch.uint8, device=device)


def _check_variant_flags(f):
    if f & ~_abi.RDN_FLAG_VARIANTS:
        raise ValueError(f"variant_flags 0x{f:x}: only the variant bits are accepted")


def _fill_fwd(a, q, k, v, g, beta, gamma, clip, S0, R0, o, ST, RT, Sc, Rc, scale, flags=0,
              cu_seqlens=None):
    B, T, H, Dk = q.shape
    a.B, a.T, a.H, a.Dk, a.Dv = B, T, H, Dk, v.shape[-1]
    a.dtype = _dtype_code(q)
    a.q, a.k, a.v = _ptr(q), _ptr(k), _ptr(v)
    a.g, a.beta, a.gamma = _ptr(g), _ptr(beta), _ptr(gamma)
    a.clip = float(clip)
    a.S0, a.R0 = _ptr(S0), _ptr(R0)
    a.o = _ptr(o)
    a.ST, a.RT = _ptr(ST), _ptr(RT)
    a.S_chunks, a.R_chunks = _ptr(Sc), _ptr(Rc)
    a.scale = float(scale)
    a.flags = flags
    if cu_seqlens is not None:
        if cu_seqlens.dtype != torch.int32 or cu_seqlens.dim() != 1 or cu_seqlens.numel() < 2:
            raise ValueError("cu_seqlens must be a 1-D int32 tensor of num_seqs + 1 offsets")
        a.cu_seqlens = _ptr(cu_seqlens)
        a.num_seqs = cu_seqlens.numel() - 1


def _num_seqs(q, cu_seqlens):
    return q.shape[0] if cu_seqlens is None else cu_seqlens.numel() - 1


def _chunk_slots(a):
    """Dk x Dv blocks in each of S_chunks and R_chunks for the filled FwdArgs."""
    n = ctypes.c_longlong(0)
    _check("rdn_chunk_slots", _abi.load().rdn_chunk_slots(ctypes.byref(a), ctypes.byref(n)))
    return n.value


def _fwd(name, q, k, v, g, beta, gamma, clip=1.0, S0=None, R0=None, scale=1.0,
         return_final_state=True, return_chunk_states=False, out=None, workspace=None,
         save_for_bwd=False, tied_gamma=False, cu_seqlens=None, variant_flags=0, f32_out=False,
         qk_norm=False, qk_eps=1e-12):
    lib = _abi.load()
    _check_variant_flags(variant_flags)
    B, T, H, Dk = q.shape
    Dv = v.shape[-1]
    dev = q.device
    N = _num_seqs(q, cu_seqlens)
    odt = torch.float32 if f32_out else q.dtype
    o = out if out is not None else torch.empty(B, T, H, Dv, dtype=odt, device=dev)
    ST = RT = Sc = Rc = None
    if return_final_state:
        ST = torch.empty(N, H, Dk, Dv, dtype=torch.float32, device=dev)
        RT = torch.empty_like(ST)
    flags = (_abi.RDN_FLAG_SAVE_FOR_BWD if save_for_bwd else 0) \
        | (_abi.RDN_FLAG_TIED_GAMMA if tied_gamma else 0) | variant_flags \
        | (_abi.RDN_FLAG_F32_OUT if f32_out else 0) | (_abi.RDN_FLAG_QK_NORM if qk_norm else 0)
    a = FwdArgs()
    _fill_fwd(a, q, k, v, g, beta, gamma, clip, S0, R0, o, ST, RT, None, None, scale, flags,
              cu_seqlens)
    a.qk_eps = float(qk_eps)
    if return_chunk_states:
        if cu_seqlens is None:
            NC = (T + CHUNK - 1) // CHUNK
            Sc = torch.empty(B, H, NC, Dk, Dv, dtype=torch.float32, device=dev)
        else:  # record slots (the packed layout of rdn_fwd_args.cu_seqlens)
            Sc = torch.empty(_chunk_slots(a), Dk, Dv, dtype=torch.float32, device=dev)
        Rc = torch.empty_like(Sc)
        a.S_chunks, a.R_chunks = _ptr(Sc), _ptr(Rc)
    nbytes = ctypes.c_size_t(0)
    _check(name + "_workspace_size",
           getattr(lib, name + "_workspace_size")(ctypes.byref(a), ctypes.byref(nbytes)))
    ws = workspace
    if ws is None or ws.numel() < nbytes.value:
        ws = _alloc_ws(nbytes.value, dev)
    a.workspace = _ptr(ws)
    a.workspace_bytes = nbytes.value if ws is not None else 0
    _check(name, getattr(lib, name)(ctypes.byref(a), _stream(q)))
    res = [o]
    if return_final_state:
        res += [ST, RT]
    if return_chunk_states:
        res += [Sc, Rc]
    return tuple(res) if len(res) > 1 else o


def rla_fwd(q, k, v, g, beta, gamma, clip=1.0, S0=None, R0=None, scale=1.0, **kw):
    """RLA forward (Section 3.4, left).  Returns (o, ST, RT)."""
    return _fwd("rla_fwd", q, k, v, g, beta, gamma, clip, S0, R0, scale, **kw)


def rdn_fwd(q, k, v, g, beta, gamma, clip=1.0, S0=None, R0=None, scale=1.0, **kw):
    """RDN forward (Section 3.4, right).  Returns (o, ST, RT) and, with
    return_chunk_states=True, also the chunk-start states (Sc, Rc) that
    rdn_bwd can reuse.  With save_for_bwd=True (needs return_chunk_states and
    a caller workspace sized with the same flag) the workspace also keeps the
    intermediates rdn_bwd(fwd_workspace=..., fwd_saved=True) reads.

    cu_seqlens (int32 device tensor of N+1 offsets, q of shape [1,T,H,D]):
    N packed sequences, each with its own recurrence; S0, R0, ST, RT are then
    [N,H,D,D] and the chunk states [slots,D,D] (rdn_fwd_args.cu_seqlens).

    qk_norm: q and k are the raw projections x; the library applies
    y = SiLU(x) / max(||SiLU(x)||, qk_eps) per row first (RDN_FLAG_QK_NORM;
    the backward takes the same keywords and returns dq, dk w.r.t. x)."""
    return _fwd("rdn_fwd", q, k, v, g, beta, gamma, clip, S0, R0, scale, **kw)


def rdn_bwd(q, k, v, g, beta, gamma, dO, clip=1.0, S0=None, R0=None, dST=None, dRT=None,
            scale=1.0, S_chunks=None, R_chunks=None, workspace=None, out=None,
            fwd_workspace=None, fwd_saved=False, tied_gamma=False, cu_seqlens=None,
            variant_flags=0, f32_out=False, qk_norm=False, qk_eps=1e-12):
    """Backward of rdn_fwd.  Returns a dict with dq, dk, dv (input dtype),
    dg (w.r.t. the log-decay), dbeta, dgamma (fp32), dS0, dR0 (fp32).

    S_chunks/R_chunks: the forward's chunk-start states (return_chunk_states).
    fwd_workspace: with them, the workspace that forward call used, whose
    per-chunk matrices are then reused instead of recomputed.
    fwd_saved: that forward ran with save_for_bwd=True.
    f32_out: dq, dk, dv in fp32 for bf16 inputs (RDN_FLAG_F32_OUT); the
    forward takes the same keyword for o.
    qk_norm, qk_eps: as given to the forward (RDN_FLAG_QK_NORM): q, k are the
    raw x and dq, dk are returned w.r.t. x."""
    return _bwd("rdn_bwd", q, k, v, g, beta, gamma, dO, clip, S0, R0, dST, dRT, scale, S_chunks,
                R_chunks, workspace, out, fwd_workspace, fwd_saved, tied_gamma, cu_seqlens,
                variant_flags, f32_out, qk_norm, qk_eps)


def rla_bwd(q, k, v, g, beta, gamma, dO, clip=1.0, S0=None, R0=None, dST=None, dRT=None,
            scale=1.0, S_chunks=None, R_chunks=None, workspace=None, out=None,
            fwd_workspace=None, fwd_saved=False, tied_gamma=False, cu_seqlens=None,
            variant_flags=0, f32_out=False, qk_norm=False, qk_eps=1e-12):
    """Backward of rla_fwd; the same arguments and results as rdn_bwd."""
    return _bwd("rla_bwd", q, k, v, g, beta, gamma, dO, clip, S0, R0, dST, dRT, scale, S_chunks,
                R_chunks, workspace, out, fwd_workspace, fwd_saved, tied_gamma, cu_seqlens,
                variant_flags, f32_out, qk_norm, qk_eps)


def _bwd(name, q, k, v, g, beta, gamma, dO, clip, S0, R0, dST, dRT, scale, S_chunks, R_chunks,
         workspace, out, fwd_workspace, fwd_saved, tied_gamma=False, cu_seqlens=None,
         variant_flags=0, f32_out=False, qk_norm=False, qk_eps=1e-12):
    lib = _abi.load()
    _check_variant_flags(variant_flags)
    B, T, H, Dk = q.shape
    Dv = v.shape[-1]
    dev = q.device
    N = _num_seqs(q, cu_seqlens)
    if out is None:
        gdt = torch.float32 if f32_out else q.dtype
        out = dict(dq=torch.empty_like(q, dtype=gdt), dk=torch.empty_like(k, dtype=gdt),
                   dv=torch.empty_like(v, dtype=gdt),
                   dg=torch.empty(B, T, H, dtype=torch.float32, device=dev),
                   dbeta=torch.empty(B, T, H, dtype=torch.float32, device=dev),
                   dgamma=torch.empty(B, T, H, dtype=torch.float32, device=dev),
                   dS0=torch.empty(N, H, Dk, Dv, dtype=torch.float32, device=dev),
                   dR0=torch.empty(N, H, Dk, Dv, dtype=torch.float32, device=dev))
    a = BwdArgs()
    _fill_fwd(a.fwd, q, k, v, g, beta, gamma, clip, S0, R0, None, None, None, S_chunks,
              R_chunks, scale, 0, cu_seqlens)
    if fwd_workspace is not None:
        a.fwd.workspace = _ptr(fwd_workspace)
        a.fwd.workspace_bytes = fwd_workspace.numel() * fwd_workspace.element_size()
    a.fwd.flags = (_abi.RDN_FLAG_SAVE_FOR_BWD if fwd_saved else 0) \
        | (_abi.RDN_FLAG_TIED_GAMMA if tied_gamma else 0) | variant_flags \
        | (_abi.RDN_FLAG_F32_OUT if f32_out else 0) | (_abi.RDN_FLAG_QK_NORM if qk_norm else 0)
    a.fwd.qk_eps = float(qk_eps)
    a.dO, a.dST, a.dRT = _ptr(dO), _ptr(dST), _ptr(dRT)
    a.dq, a.dk, a.dv = _ptr(out["dq"]), _ptr(out["dk"]), _ptr(out["dv"])
    a.dg, a.dbeta, a.dgamma = _ptr(out["dg"]), _ptr(out["dbeta"]), _ptr(out.get("dgamma"))
    a.dS0, a.dR0 = _ptr(out.get("dS0")), _ptr(out.get("dR0"))
    nbytes = ctypes.c_size_t(0)
    _check(name + "_workspace_size",
           getattr(lib, name + "_workspace_size")(ctypes.byref(a), ctypes.byref(nbytes)))
    ws = workspace
    if ws is None or ws.numel() < nbytes.value:
        ws = _alloc_ws(nbytes.value, dev)
    a.workspace = _ptr(ws)
    a.workspace_bytes = nbytes.value if ws is not None else 0
    _check(name, getattr(lib, name)(ctypes.byref(a), _stream(q)))
    return out


def _prologue_args(x0, x1, eps):
    a = _abi.PrologueArgs()
    D = x0.shape[-1]
    a.rows = x0.numel() // D
    a.D = D
    a.dtype = _dtype_code(x0)
    a.eps = float(eps)
    a.x[0], a.x[1] = _ptr(x0), _ptr(x1)
    if x1 is not None and x1.shape != x0.shape:
        raise ValueError("q and k must have the same shape")
    return a


def qk_prologue(q, k=None, eps=1e-12, out=None):
    """SiLU then L2 normalisation over the last axis, of q and (optionally) k
    in one launch: y = SiLU(x) / max(||SiLU(x)||, eps).  Returns (q', k') (k'
    None when k is None)."""
    lib = _abi.load()
    yq = out[0] if out is not None else torch.empty_like(q)
    yk = (out[1] if out is not None else torch.empty_like(k)) if k is not None else None
    a = _prologue_args(q, k, eps)
    a.y[0], a.y[1] = _ptr(yq), _ptr(yk)
    _check("rdn_qk_prologue", lib.rdn_qk_prologue(ctypes.byref(a), _stream(q)))
    return yq, yk


def qk_prologue_bwd(q, k, dyq, dyk=None, eps=1e-12, out=None):
    """Gradients w.r.t. the pre-activation q, k of <dyq, q'> + <dyk, k'>
    (q', k' from qk_prologue; recomputed from q, k).  k / dyk may be None;
    out: (dq, dk) buffers to write into."""
    lib = _abi.load()
    if out is not None:
        dq, dk = out
    else:
        dq = torch.empty_like(q)
        dk = torch.empty_like(k) if k is not None else None
    a = _prologue_args(q, k, eps)
    a.dy[0], a.dy[1] = _ptr(dyq), _ptr(dyk)
    a.dx[0], a.dx[1] = _ptr(dq), _ptr(dk)
    _check("rdn_qk_prologue_bwd", lib.rdn_qk_prologue_bwd(ctypes.byref(a), _stream(q)))
    return dq, dk


def rdn_decode_step(q, k, v, g, beta, gamma, S, R, clip=1.0, scale=1.0, variant="rdn", out=None,
                    tied_gamma=False, variant_flags=0, qk_norm=False, qk_eps=1e-12):
    """One recurrent step for N sequences; S, R [N,H,Dk,Dv] fp32 are updated
    in place.  q, k [N,H,Dk]; v [N,H,Dv]; gates [N,H].  Returns o [N,H,Dv].
    tied_gamma / variant_flags / qk_norm, qk_eps: as for the forward."""
    lib = _abi.load()
    _check_variant_flags(variant_flags)
    N, H, Dk = q.shape
    Dv = v.shape[-1]
    o = out if out is not None else torch.empty(N, H, Dv, dtype=q.dtype, device=q.device)
    a = DecodeArgs()
    a.N, a.H, a.Dk, a.Dv = N, H, Dk, Dv
    a.dtype = _dtype_code(q)
    a.variant = 1 if variant == "rdn" else 0
    a.q, a.k, a.v = _ptr(q), _ptr(k), _ptr(v)
    a.g, a.beta, a.gamma = _ptr(g), _ptr(beta), _ptr(gamma)
    a.clip, a.scale = float(clip), float(scale)
    a.S, a.R, a.o = _ptr(S), _ptr(R), _ptr(o)
    a.flags = (_abi.RDN_FLAG_TIED_GAMMA if tied_gamma else 0) | variant_flags \
        | (_abi.RDN_FLAG_QK_NORM if qk_norm else 0)
    a.qk_eps = float(qk_eps)
    _check("rdn_decode_step", lib.rdn_decode_step(ctypes.byref(a), _stream(q)))
    return o


def device_status(stream=None):
    """Wait for the stream (default: torch's current stream) and return the
    device-side failure code recorded since the last call (0 = none; 4 = a
    bounded wait gave up, the outputs of that call are invalid), clearing it."""
    st = ctypes.c_int(0)
    s = torch.cuda.current_stream().cuda_stream if stream is None else stream.cuda_stream
    _check("rdn_device_status", _abi.load().rdn_device_status(s, ctypes.byref(st)))
    return st.value


class LaunchTimer:
    """Context manager recording the device time of every launch of the
    library's kernels (CUDA events on each kernel's own stream).

        with LaunchTimer() as lt:
            ...
        lt.records  -> [(kernel_name, ms), ...];  lt.launches -> count"""

    def __init__(self, capacity=65536):
        self.capacity = capacity
        self.records = []
        self.launches = 0

    def __enter__(self):
        _check("rdn_prof_start", _abi.load().rdn_prof_start(self.capacity))
        return self

    def __exit__(self, *exc):
        buf = (_abi.ProfRecord * self.capacity)()
        n = ctypes.c_int(0)
        _check("rdn_prof_stop", _abi.load().rdn_prof_stop(buf, self.capacity, ctypes.byref(n)))
        self.launches = n.value
        self.records = [(buf[i].name.decode(), float(buf[i].ms))
                        for i in range(min(n.value, self.capacity))]
        return False

    def summary(self):
        """{kernel: (launches, total_ms, mean_ms)}"""
        out = {}
        for name, ms in self.records:
            c, t = out.get(name, (0, 0.0))[:2]
            out[name] = (c + 1, t + ms)
        return {k: (c, t, t / c) for k, (c, t) in out.items()}


def workspace_bytes(op, B, T, H, D, dtype=torch.bfloat16, save_for_bwd=False, cu_seqlens=None,
                    variant_flags=0, qk_norm=False):
    """Workspace size the library asks for (op: rla_fwd | rdn_fwd | rla_bwd | rdn_bwd);
    cu_seqlens: the packed-sequence table of the call (B = 1); variant_flags:
    the variant bits of the call; qk_norm: the call normalises q, k."""
    lib = _abi.load()
    a = FwdArgs()
    a.B, a.T, a.H, a.Dk, a.Dv = B, T, H, D, D
    a.dtype = _abi.RDN_BF16 if dtype == torch.bfloat16 else _abi.RDN_F32
    a.clip, a.scale = 1.0, 1.0
    _check_variant_flags(variant_flags)
    a.flags = (_abi.RDN_FLAG_SAVE_FOR_BWD if save_for_bwd else 0) | variant_flags \
        | (_abi.RDN_FLAG_QK_NORM if qk_norm else 0)
    a.qk_eps = 1e-12
    if cu_seqlens is not None:
        a.cu_seqlens, a.num_seqs = _ptr(cu_seqlens), cu_seqlens.numel() - 1
    n = ctypes.c_size_t(0)
    if op in ("rla_bwd", "rdn_bwd"):
        b = BwdArgs()
        b.fwd = a
        _check(op, getattr(lib, op + "_workspace_size")(ctypes.byref(b), ctypes.byref(n)))
    else:
        _check(op, getattr(lib, op + "_workspace_size")(ctypes.byref(a), ctypes.byref(n)))
    return n.value
