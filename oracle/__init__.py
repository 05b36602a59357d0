"""fp64 CPU oracle for RLA / RDN (arXiv 2509.25223), Section 3.4.

TEST INFRASTRUCTURE ONLY.  Only ``tests/``, ``__graft_entry__.smoke()`` and
the CPU-baseline / reference leg of ``bench.py`` may import this package.
The product library (``paper_2509_25223_gb300``) never imports it and shares
no code with it; the two meet only in the seeded input generator
(``rdn_synthetic``), which holds none of the method's arithmetic.

The arithmetic lives in ``rdn_oracle.c``: the paper's token recurrence
(Section 3.4, "Final Formulations"; clipping Section 3.3) written out one token
at a time in double precision, plus hand-written back-propagation through
time.  This module compiles it with gcc (``build()``) and wraps it with ctypes.
All arrays are numpy float64, C-contiguous, in the layouts

    q, k [B,T,H,Dk]   v, o [B,T,H,Dv]   g, beta, gamma [B,T,H]
    S0, R0, ST, RT [B,H,Dk,Dv]

where g = log(alpha) is the per-token log-decay and the states are stored
[d_k][d_v] (the paper's d_v x d_k matrices, transposed).
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "rdn_oracle.c")
_BUILD_DIR = os.path.join(_HERE, "_build")
_SO = os.path.join(_BUILD_DIR, "liboracle.so")
_lock = threading.Lock()
_lib = None

RLA, RDN = 0, 1
# variant bits (rdn_oracle.c, orc_fwd_mod): residual against a_t S_{t-1} k_t;
# ungated combine o = S_{t-1} q + R_t q; c tanh(x / c) residual; stateless
# correction R_t = r_t k_t^T
DECAYED, PLAIN, TANH, STATELESS = 1, 2, 4, 8


def build(force: bool = False) -> str:
    """Compile rdn_oracle.c into oracle/_build/liboracle.so (gcc, OpenMP).

    -ffp-contract=off keeps x86_64 and aarch64 results bit-identical."""
    os.makedirs(_BUILD_DIR, exist_ok=True)
    if force or not os.path.exists(_SO) or os.path.getmtime(_SO) < os.path.getmtime(_SRC):
        tmp = _SO + f".tmp{os.getpid()}"
        cmd = ["gcc", "-O3", "-ffp-contract=off", "-fopenmp", "-fPIC", "-shared",
               "-std=c11", "-o", tmp, _SRC, "-lm"]
        subprocess.run(cmd, check=True)
        os.replace(tmp, _SO)
    return _SO


def _load():
    global _lib
    with _lock:
        if _lib is None:
            lib = ctypes.CDLL(build())
            P = ctypes.c_void_p
            I = ctypes.c_int
            D = ctypes.c_double
            fwd_sig = [I, I, I, I, I, P, P, P, P, P, P, D, D, P, P, P, P, P]
            for name in ("orc_rla_fwd", "orc_rdn_fwd"):
                getattr(lib, name).argtypes = fwd_sig
                getattr(lib, name).restype = None
            lib.orc_fwd_mod.argtypes = [I, I] + fwd_sig + [P]
            lib.orc_fwd_mod.restype = None
            bwd_sig = [I, I, I, I, I, P, P, P, P, P, P, D, D, P, P, P, P, P,
                       P, P, P, P, P, P, P, P]
            for name in ("orc_rla_bwd", "orc_rdn_bwd"):
                getattr(lib, name).argtypes = bwd_sig
                getattr(lib, name).restype = None
            lib.orc_bwd_mod.argtypes = [I, I] + bwd_sig
            lib.orc_bwd_mod.restype = None
            lib.orc_decode_step.argtypes = [I, I, I, I, I, P, P, P, P, P, P, D, D, P, P, P]
            lib.orc_decode_step.restype = None
            lib.orc_clip_margin_condition.argtypes = [I, I, I, I, I, I, P, P, P, P, P, P,
                                                      D, D, P, P, D, I, I]
            lib.orc_clip_margin_condition.restype = ctypes.c_long
            lib.orc_max_threads.restype = I
            lib.orc_set_threads.argtypes = [I]
            _lib = lib
    return _lib


def _f64(x):
    if x is None:
        return None
    if hasattr(x, "detach"):  # torch tensor
        x = x.detach().cpu().double().numpy()
    return np.ascontiguousarray(x, dtype=np.float64)


def _ptr(a):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


def max_threads() -> int:
    return _load().orc_max_threads()


def set_threads(n: int) -> None:
    _load().orc_set_threads(int(n))


def _dims(q, v):
    B, T, H, Dk = q.shape
    Dv = v.shape[-1]
    return B, T, H, Dk, Dv


def fwd(variant, q, k, v, g, beta, gamma, c=1.0, S0=None, R0=None, scale=1.0,
        return_residual=False, mods=0):
    """Forward of RLA (variant=RLA) or RDN (variant=RDN), with the variant
    bits `mods` (DECAYED | PLAIN | TANH | STATELESS, 0 = the method).

    Returns (o, ST, RT) as float64 arrays, plus r (the clipped residuals,
    [B,T,H,Dv]) when return_residual is set."""
    lib = _load()
    q, k, v, g, beta, gamma = map(_f64, (q, k, v, g, beta, gamma))
    S0, R0 = _f64(S0), _f64(R0)
    B, T, H, Dk, Dv = _dims(q, v)
    o = np.zeros((B, T, H, Dv))
    ST = np.zeros((B, H, Dk, Dv))
    RT = np.zeros((B, H, Dk, Dv))
    args = (B, T, H, Dk, Dv, _ptr(q), _ptr(k), _ptr(v), _ptr(g), _ptr(beta),
            _ptr(gamma), float(c), float(scale), _ptr(S0), _ptr(R0), _ptr(o),
            _ptr(ST), _ptr(RT))
    if return_residual or mods:
        r = np.zeros((B, T, H, Dv)) if return_residual else None
        lib.orc_fwd_mod(int(variant), int(mods), *args, _ptr(r))
        return (o, ST, RT, r) if return_residual else (o, ST, RT)
    (lib.orc_rdn_fwd if variant == RDN else lib.orc_rla_fwd)(*args)
    return o, ST, RT


def rdn_fwd(*a, **kw):
    """RDN forward (Section 3.4, right formulation)."""
    return fwd(RDN, *a, **kw)


def rla_fwd(*a, **kw):
    """RLA forward (Section 3.4, left formulation)."""
    return fwd(RLA, *a, **kw)


def bwd(variant, q, k, v, g, beta, gamma, c, S0, R0, dO, dST=None, dRT=None,
        scale=1.0, mods=0):
    """Back-propagation through time of the forward above.

    Returns a dict with dq, dk, dv, dg (w.r.t. the log-decay g), dbeta,
    dgamma, dS0, dR0 (float64)."""
    lib = _load()
    q, k, v, g, beta, gamma, dO = map(_f64, (q, k, v, g, beta, gamma, dO))
    S0, R0, dST, dRT = map(_f64, (S0, R0, dST, dRT))
    B, T, H, Dk, Dv = _dims(q, v)
    out = dict(dq=np.zeros((B, T, H, Dk)), dk=np.zeros((B, T, H, Dk)),
               dv=np.zeros((B, T, H, Dv)), dg=np.zeros((B, T, H)),
               dbeta=np.zeros((B, T, H)), dgamma=np.zeros((B, T, H)),
               dS0=np.zeros((B, H, Dk, Dv)), dR0=np.zeros((B, H, Dk, Dv)))
    fn = lib.orc_rdn_bwd if variant == RDN else lib.orc_rla_bwd
    if mods:
        fn = lambda *a: lib.orc_bwd_mod(int(variant), int(mods), *a)  # noqa: E731
    fn(B, T, H, Dk, Dv, _ptr(q), _ptr(k), _ptr(v), _ptr(g), _ptr(beta),
       _ptr(gamma), float(c), float(scale), _ptr(S0), _ptr(R0), _ptr(dO),
       _ptr(dST), _ptr(dRT), _ptr(out["dq"]), _ptr(out["dk"]), _ptr(out["dv"]),
       _ptr(out["dg"]), _ptr(out["dbeta"]), _ptr(out["dgamma"]),
       _ptr(out["dS0"]), _ptr(out["dR0"]))
    return out


def rdn_bwd(*a, **kw):
    return bwd(RDN, *a, **kw)


def rla_bwd(*a, **kw):
    return bwd(RLA, *a, **kw)


def decode_step(variant, q, k, v, g, beta, gamma, c, S, R, scale=1.0):
    """One recurrent step for N independent sequences.

    q, k [N,H,Dk]; v [N,H,Dv]; gates [N,H]; S, R [N,H,Dk,Dv].
    Returns (o [N,H,Dv], S_new, R_new); the inputs are not modified."""
    lib = _load()
    q, k, v, g, beta, gamma = map(_f64, (q, k, v, g, beta, gamma))
    S = _f64(S).copy()
    R = _f64(R).copy()
    N, H, Dk = q.shape
    Dv = v.shape[-1]
    o = np.zeros((N, H, Dv))
    lib.orc_decode_step(int(variant), N, H, Dk, Dv, _ptr(q), _ptr(k), _ptr(v),
                        _ptr(g), _ptr(beta), _ptr(gamma), float(c), float(scale),
                        _ptr(S), _ptr(R), _ptr(o))
    return o, S, R


# ----------------------------------------------------------- q, k prologue
# Section 3.4 leaves out of its equations the SiLU activation and the L2
# normalisation that the model applies to queries and keys before the
# recurrence; the reading here: SiLU first, then normalisation over the head
# dimension, with the norm floored at eps like the listing's normalisation.

def qk_prologue(x, eps=1e-12):
    """y = u / max(||u||_2, eps), u = SiLU(x) = x * sigmoid(x), over the last
    axis of x (rows of q or k, [..., D])."""
    x = _f64(x)
    u = x / (1.0 + np.exp(-x))
    n = np.sqrt((u * u).sum(-1, keepdims=True))
    return u / np.maximum(n, eps)


def qk_prologue_bwd(x, dy, eps=1e-12):
    """Gradient of <dy, qk_prologue(x)> w.r.t. x, by the chain rule through the
    two steps: with y = u / n (n = ||u|| > eps) du = (dy - y <y, dy>) / n, with
    n <= eps du = dy / eps; then dx = du * SiLU'(x), SiLU'(x) = s (1 + x (1 - s)),
    s = sigmoid(x)."""
    x, dy = _f64(x), _f64(dy)
    s = 1.0 / (1.0 + np.exp(-x))
    u = x * s
    n = np.sqrt((u * u).sum(-1, keepdims=True))
    big = n > eps
    y = u / np.maximum(n, eps)
    du = np.where(big, (dy - y * (y * dy).sum(-1, keepdims=True)) / np.maximum(n, eps), dy / eps)
    return du * s * (1.0 + x * (1.0 - s))


QUANT = {"f64": 0, "f32": 1, "bf16": 2}


def _bf16_tie_distance(y):
    """|position of y between its two neighbouring bf16 values - 1/2|, in
    units of that spacing (0 = exactly halfway, 1/2 = on a bf16 value)."""
    a = np.abs(y)
    e = np.floor(np.log2(np.maximum(a, np.finfo(np.float32).tiny)))
    ulp = np.exp2(e - 7.0)  # 8 significant bits
    f = a / ulp - np.floor(a / ulp)
    return np.abs(f - 0.5)


def qk_round_margin_condition(x, eps=1e-12, margin=2.0 ** -9, max_iter=64):
    """Return (x_conditioned, n_moved): bf16 rows x [..., D] moved, one bf16
    step at a time, so that every element of the fp64 prologue output y (as
    qk_prologue computes it) is at least `margin` bf16 spacings away from a
    rounding tie of bf16.  A library that holds y in bf16 after computing it
    in fp32 (relative error well below 2^-17, i.e. 2^-9 of a bf16 spacing)
    then rounds every y to the bf16 value that the fp64 y rounds to, so the
    reference and the library see the same y.  In a row with an element too
    close to a tie the element of largest SiLU(x) among those that are not
    takes one bf16 step up (SiLU rises there with slope about 1, so the row's
    norm, and with it every y of the row, moves by a fraction of a spacing;
    stepping an element near a tie would move its own y by about one spacing
    and keep it there); rows are revisited until none is left."""
    x = _f64(x).copy()
    D = x.shape[-1]
    flat = x.reshape(-1, D)
    moved = 0

    def silu(rows):
        return flat[rows] / (1.0 + np.exp(-flat[rows]))

    def near(rows):
        u = silu(rows)
        n = np.sqrt((u * u).sum(-1, keepdims=True))
        return _bf16_tie_distance(u / np.maximum(n, eps)) < margin

    rows = np.arange(flat.shape[0])
    rows = rows[near(rows).any(-1)]
    for _ in range(max_iter):
        if rows.size == 0:
            break
        j = np.where(near(rows), -np.inf, silu(rows)).argmax(-1)
        v = flat[rows, j]
        a = np.maximum(np.abs(v), np.finfo(np.float32).tiny)
        # one bf16 step up: the spacing above v (below a power of two going
        # down from a negative v it is half as large, a finer step, also fine)
        flat[rows, j] = v + np.exp2(np.floor(np.log2(a)) - 7.0)
        moved += rows.size
        rows = rows[near(rows).any(-1)]
    if rows.size:
        raise RuntimeError(f"qk_round_margin_condition: {rows.size} rows left near a tie")
    return flat.reshape(x.shape), moved


def clip_margin_condition(variant, q, k, v, g, beta, gamma, c, S0=None, R0=None,
                          scale=1.0, margin=4e-3, quant="bf16", mods=0):
    """Return (v_conditioned, n_moved): v moved, in token order and in steps
    representable in `quant`, so that every |v - S_{t-1}k| of the fp64
    forward is at least `margin` away from the clip threshold c.  Makes the
    clip mask, and so the backward, unique at tolerance level."""
    lib = _load()
    q, k, g, beta, gamma = map(_f64, (q, k, g, beta, gamma))
    v = _f64(v).copy()
    S0, R0 = _f64(S0), _f64(R0)
    B, T, H, Dk, Dv = _dims(q, v)
    n = lib.orc_clip_margin_condition(int(variant), B, T, H, Dk, Dv, _ptr(q), _ptr(k),
                                      _ptr(v), _ptr(g), _ptr(beta), _ptr(gamma),
                                      float(c), float(scale), _ptr(S0), _ptr(R0),
                                      float(margin), QUANT[quant], int(mods))
    return v, int(n)
