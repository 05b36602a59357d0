"""The C-ABI library: builds, loads, exports what include/rdn.h declares, and
rejects bad arguments with a status code before touching the GPU (CPU only)."""
import ctypes
import math
import os
import re
import subprocess

import pytest

import paper_2509_25223_gb300 as rdn
from paper_2509_25223_gb300 import _abi

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _header_functions():
    src = open(os.path.join(ROOT, "include", "rdn.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"^\s*(?:const\s+)?\w+\s*\*?\s*(\w+)\s*\(", src, flags=re.M)))


def test_header_matches_binding():
    assert _header_functions() == sorted(_abi.EXPORTS)


def test_library_exports_every_declared_symbol():
    lib = _abi.load()
    out = subprocess.run(["nm", "-D", "--defined-only", _abi.lib_path()], capture_output=True,
                         text=True, check=True).stdout
    exported = {ln.split()[-1] for ln in out.splitlines() if ln.strip()}
    for name in _header_functions():
        assert name in exported, name
        assert getattr(lib, name) is not None
    assert lib.rdn_version().decode().startswith("rdn-gb300")


def _fwd_args(**over):
    a = _abi.FwdArgs()
    a.B, a.T, a.H, a.Dk, a.Dv = 2, 128, 4, 128, 128
    a.dtype = _abi.RDN_BF16
    a.clip, a.scale = 1.0, 1.0
    for k, v in over.items():
        setattr(a, k, v)
    return a


def _status(fn, a):
    lib = _abi.load()
    return getattr(lib, fn)(ctypes.byref(a), None)


FAKE = ctypes.c_void_p(0x10000)  # aligned, never dereferenced: validation fails first


@pytest.mark.parametrize("fn", ["rla_fwd", "rdn_fwd"])
def test_fwd_validation(fn):
    lib = _abi.load()
    assert lib[fn](None, None) == 1
    assert _status(fn, _fwd_args(B=0)) == 1
    assert _status(fn, _fwd_args(T=-1)) == 1
    assert _status(fn, _fwd_args(Dk=96, Dv=96)) == 2
    assert _status(fn, _fwd_args(Dk=128, Dv=64)) == 2
    assert _status(fn, _fwd_args(dtype=7)) == 2
    assert _status(fn, _fwd_args(clip=-1.0)) == 1
    assert _status(fn, _fwd_args(clip=float("nan"))) == 1
    assert _status(fn, _fwd_args(flags=0x100)) == 2
    # q, k normalisation: needs a positive finite floor; then the NULL check
    QKN = _abi.RDN_FLAG_QK_NORM
    assert _status(fn, _fwd_args(flags=QKN)) == 1
    assert "qk_eps" in lib.rdn_last_error().decode()
    assert _status(fn, _fwd_args(flags=QKN, qk_eps=float("inf"))) == 1
    assert _status(fn, _fwd_args(flags=QKN, qk_eps=1e-12)) == 1
    assert "q is NULL" in lib.rdn_last_error().decode()
    # fp32 results: bf16 inputs need the tensor-core path (Dk = 128); fp32
    # inputs take the flag as a no-op (then the call
    # gets as far as the NULL pointer check)
    F32 = _abi.RDN_FLAG_F32_OUT
    assert _status(fn, _fwd_args(flags=F32, Dk=64, Dv=64)) == 2
    assert _status(fn, _fwd_args(flags=F32 | _abi.RDN_FLAG_TANH_RESIDUAL)) == 1
    assert _status(fn, _fwd_args(flags=F32 | _abi.RDN_FLAG_STATELESS_AUX)) == 1
    assert _status(fn, _fwd_args(flags=F32)) == 1
    assert _status(fn, _fwd_args(flags=F32 | _abi.RDN_FLAG_DECAYED_RESIDUAL)) == 1
    assert _status(fn, _fwd_args(flags=F32, dtype=_abi.RDN_F32, Dk=64, Dv=64)) == 1
    # tied gates: gamma may be NULL (beta serves as both); the call then gets
    # as far as the workspace check
    tied = dict(q=FAKE, k=FAKE, v=FAKE, g=FAKE, beta=FAKE, o=FAKE)
    assert _status(fn, _fwd_args(flags=_abi.RDN_FLAG_TIED_GAMMA, **tied)) == 5
    assert _status(fn, _fwd_args(flags=0, **tied)) == 1  # untied: gamma is required
    # RDN_FLAG_SAVE_FOR_BWD: only with chunk states
    assert _status(fn, _fwd_args(flags=_abi.RDN_FLAG_SAVE_FOR_BWD)) == 1  # needs S_chunks
    assert _status(fn, _fwd_args()) == 1  # q is NULL
    assert "q is NULL" in lib.rdn_last_error().decode()
    ok = dict(q=FAKE, k=FAKE, v=FAKE, g=FAKE, beta=FAKE, gamma=FAKE, o=FAKE)
    mis = dict(ok)
    mis["v"] = ctypes.c_void_p(0x10004)
    assert _status(fn, _fwd_args(**mis)) == 6
    assert _status(fn, _fwd_args(S_chunks=FAKE, **ok)) == 1  # R_chunks missing
    if fn == "rdn_fwd":
        assert _status(fn, _fwd_args(flags=_abi.RDN_FLAG_SAVE_FOR_BWD, **ok)) == 1
        assert "S_chunks" in lib.rdn_last_error().decode()
    assert _status(fn, _fwd_args(**ok)) == 5  # no workspace
    assert "workspace" in lib.rdn_last_error().decode()


def test_workspace_size_queries():
    lib = _abi.load()
    n = ctypes.c_size_t(0)
    assert lib.rdn_fwd_workspace_size(ctypes.byref(_fwd_args()), ctypes.byref(n)) == 0
    assert n.value > 0
    assert lib.rdn_fwd_workspace_size(ctypes.byref(_fwd_args(Dk=32, Dv=32)), ctypes.byref(n)) == 2
    assert lib.rdn_fwd_workspace_size(ctypes.byref(_fwd_args()), None) == 1
    m = ctypes.c_size_t(0)
    a = _fwd_args(flags=_abi.RDN_FLAG_SAVE_FOR_BWD)
    assert lib.rdn_fwd_workspace_size(ctypes.byref(a), ctypes.byref(m)) == 0
    # E, E2 (fp32 [64][Dv] each) and the mask (one word per value column) per chunk
    nct = a.B * a.H * ((a.T + 63) // 64)
    assert m.value - n.value == nct * (2 * 64 * 128 * 4 + 128 * 8)


def test_packed_sequence_validation_and_sizes():
    """cu_seqlens: B must be 1, num_seqs >= 1, the table 16-byte aligned; the
    chunk-slot count and the workspace grow by H * num_seqs records."""
    lib = _abi.load()
    ok = dict(q=FAKE, k=FAKE, v=FAKE, g=FAKE, beta=FAKE, gamma=FAKE, o=FAKE)
    assert _status("rdn_fwd", _fwd_args(cu_seqlens=FAKE, num_seqs=3, **ok)) == 1  # B = 2
    assert "B = 1" in lib.rdn_last_error().decode()
    assert _status("rdn_fwd", _fwd_args(B=1, cu_seqlens=FAKE, num_seqs=0, **ok)) == 1
    assert _status("rdn_fwd", _fwd_args(B=1, cu_seqlens=ctypes.c_void_p(0x10004), num_seqs=3,
                                        **ok)) == 6
    assert _status("rdn_fwd", _fwd_args(B=1, cu_seqlens=FAKE, num_seqs=3, **ok)) == 5
    slots = ctypes.c_longlong(0)
    a = _fwd_args(B=1, T=300, H=4)
    assert lib.rdn_chunk_slots(ctypes.byref(a), ctypes.byref(slots)) == 0
    assert slots.value == 4 * 5
    p = _fwd_args(B=1, T=300, H=4, cu_seqlens=FAKE, num_seqs=7)
    assert lib.rdn_chunk_slots(ctypes.byref(p), ctypes.byref(slots)) == 0
    assert slots.value == 4 * (7 + 5)  # at most num_seqs + ceil(T/64) chunks per head
    n, m = ctypes.c_size_t(0), ctypes.c_size_t(0)
    assert lib.rdn_fwd_workspace_size(ctypes.byref(a), ctypes.byref(n)) == 0
    assert lib.rdn_fwd_workspace_size(ctypes.byref(p), ctypes.byref(m)) == 0
    rec = (n.value - 256) // (4 * 5)
    table = 256  # 8 entries of {first token, first chunk}, rounded up to 256 bytes
    assert m.value == 256 + rec * 4 * 12 + table


def test_device_status_validation():
    lib = _abi.load()
    assert lib.rdn_device_status(None, None) == 1  # status pointer NULL, before any CUDA call
    assert "status is NULL" in lib.rdn_last_error().decode()


def test_decode_validation():
    lib = _abi.load()
    a = _abi.DecodeArgs()
    a.N, a.H, a.Dk, a.Dv, a.dtype, a.variant = 4, 2, 128, 128, _abi.RDN_BF16, 1
    a.clip, a.scale = 1.0, 1.0
    assert lib.rdn_decode_step(ctypes.byref(a), None) == 1  # NULL pointers
    for f in ("q", "k", "v", "g", "beta", "gamma", "o"):
        setattr(a, f, FAKE)
    a.S = ctypes.c_void_p(0x20000)
    a.R = ctypes.c_void_p(0x20000)
    assert lib.rdn_decode_step(ctypes.byref(a), None) == 1  # S aliases R
    assert "alias" in lib.rdn_last_error().decode()
    a.variant = 3
    assert lib.rdn_decode_step(ctypes.byref(a), None) == 1
    a.variant = 1
    a.clip = -2.0
    assert lib.rdn_decode_step(ctypes.byref(a), None) == 1
    a.clip = math.inf
    a.flags = 0x40
    assert lib.rdn_decode_step(ctypes.byref(a), None) == 2  # not a variant flag
    a.flags = 0
    a.Dk = a.Dv = 256
    assert lib.rdn_decode_step(ctypes.byref(a), None) == 2


def test_bwd_validation():
    lib = _abi.load()
    b = _abi.BwdArgs()
    b.fwd = _fwd_args()
    assert lib.rdn_bwd(ctypes.byref(b), None) == 1
    b.fwd = _fwd_args(clip=-0.5)
    assert lib.rdn_bwd(ctypes.byref(b), None) == 1
    ok = dict(q=FAKE, k=FAKE, v=FAKE, g=FAKE, beta=FAKE, gamma=FAKE)
    for f in ("dO", "dq", "dk", "dv", "dg", "dbeta", "dgamma"):
        setattr(b, f, FAKE)
    # the forward's workspace is reused only with its chunk states
    b.fwd = _fwd_args(workspace=FAKE, workspace_bytes=1 << 40, **ok)
    assert lib.rdn_bwd(ctypes.byref(b), None) == 1
    assert "S_chunks" in lib.rdn_last_error().decode()
    n = ctypes.c_size_t(0)
    assert lib.rdn_fwd_workspace_size(ctypes.byref(_fwd_args()), ctypes.byref(n)) == 0
    b.fwd = _fwd_args(workspace=FAKE, workspace_bytes=n.value - 16, S_chunks=FAKE, R_chunks=FAKE,
                      **ok)
    assert lib.rdn_bwd(ctypes.byref(b), None) == 5
    assert "fwd.workspace" in lib.rdn_last_error().decode()
    b.fwd = _fwd_args(workspace=ctypes.c_void_p(0x10008), workspace_bytes=n.value, S_chunks=FAKE,
                      R_chunks=FAKE, **ok)
    assert lib.rdn_bwd(ctypes.byref(b), None) == 5
    # saved intermediates: need the forward's workspace, sized with the flag
    b.fwd = _fwd_args(flags=_abi.RDN_FLAG_SAVE_FOR_BWD, S_chunks=FAKE, R_chunks=FAKE, **ok)
    assert lib.rdn_bwd(ctypes.byref(b), None) == 1
    b.fwd = _fwd_args(flags=_abi.RDN_FLAG_SAVE_FOR_BWD, workspace=FAKE, workspace_bytes=n.value,
                      S_chunks=FAKE, R_chunks=FAKE, **ok)
    assert lib.rdn_bwd(ctypes.byref(b), None) == 5


def test_rla_bwd_validation():
    """rla_bwd shares rdn_bwd's checks, the saved-intermediates flag included
    (it needs the forward's workspace); its workspace query answers for the
    RLA forward's layout."""
    lib = _abi.load()
    b = _abi.BwdArgs()
    b.fwd = _fwd_args()
    assert lib.rla_bwd(ctypes.byref(b), None) == 1
    ok = dict(q=FAKE, k=FAKE, v=FAKE, g=FAKE, beta=FAKE, gamma=FAKE)
    for f in ("dO", "dq", "dk", "dv", "dg", "dbeta", "dgamma"):
        setattr(b, f, FAKE)
    b.fwd = _fwd_args(flags=_abi.RDN_FLAG_SAVE_FOR_BWD, S_chunks=FAKE, R_chunks=FAKE, **ok)
    assert lib.rla_bwd(ctypes.byref(b), None) == 1  # the flag without the forward's workspace
    assert "RDN_FLAG_SAVE_FOR_BWD" in lib.rdn_last_error().decode()
    n_rla, n_rdn = ctypes.c_size_t(0), ctypes.c_size_t(0)
    b.fwd = _fwd_args()
    assert lib.rla_bwd_workspace_size(ctypes.byref(b), ctypes.byref(n_rla)) == 0
    assert lib.rdn_bwd_workspace_size(ctypes.byref(b), ctypes.byref(n_rdn)) == 0
    assert n_rla.value > 0 and n_rdn.value > 0
    # the forward's workspace must be at least what rla_fwd asks for
    nf = ctypes.c_size_t(0)
    assert lib.rla_fwd_workspace_size(ctypes.byref(_fwd_args()), ctypes.byref(nf)) == 0
    b.fwd = _fwd_args(workspace=FAKE, workspace_bytes=nf.value - 16, S_chunks=FAKE, R_chunks=FAKE,
                      **ok)
    assert lib.rla_bwd(ctypes.byref(b), None) == 5


def test_binding_rejects_cpu_tensors():
    import torch
    x = torch.zeros(1, 64, 1, 64)
    g = torch.zeros(1, 64, 1)
    with pytest.raises(ValueError):
        rdn.rla_fwd(x, x, x, g, g, g)


_STRUCTS = {
    "rdn_fwd_args": ("FwdArgs", ["B", "q", "clip", "S0", "scale", "flags", "workspace",
                                 "workspace_bytes", "cu_seqlens", "num_seqs", "qk_eps"]),
    "rdn_bwd_args": ("BwdArgs", ["fwd", "dO", "dq", "dS0", "dR0", "workspace",
                                 "workspace_bytes"]),
    "rdn_decode_args": ("DecodeArgs", ["N", "variant", "q", "clip", "scale", "S", "o", "flags",
                                       "qk_eps"]),
    "rdn_prologue_args": ("PrologueArgs", ["rows", "D", "dtype", "eps", "x", "y", "dy", "dx"]),
}


def test_binding_struct_layouts_match_the_header(tmp_path):
    """sizeof and field offsets of every argument struct, as the C compiler lays
    them out from include/rdn.h, equal those of the ctypes binding."""
    src = ["#include <stdio.h>", "#include <stddef.h>", '#include "rdn.h"', "int main(void) {"]
    for cname, (_, fields) in _STRUCTS.items():
        src.append(f'  printf("{cname} size %zu\\n", sizeof({cname}));')
        for f in fields:
            src.append(f'  printf("{cname} {f} %zu\\n", offsetof({cname}, {f}));')
    src += ["  return 0;", "}"]
    c = tmp_path / "layout.c"
    c.write_text("\n".join(src))
    exe = tmp_path / "layout"
    subprocess.run(["gcc", "-I", os.path.join(ROOT, "include"), str(c), "-o", str(exe)], check=True)
    out = subprocess.run([str(exe)], capture_output=True, text=True, check=True).stdout.split("\n")
    got = {tuple(ln.split()[:2]): int(ln.split()[2]) for ln in out if ln.strip()}
    for cname, (pyname, fields) in _STRUCTS.items():
        st = getattr(_abi, pyname)
        assert got[(cname, "size")] == ctypes.sizeof(st), cname
        for f in fields:
            assert got[(cname, f)] == getattr(st, f).offset, (cname, f)


def test_binding_flag_values_match_the_header():
    """Every RDN_FLAG_* of include/rdn.h has the same value in the binding."""
    src = open(os.path.join(ROOT, "include", "rdn.h")).read()
    flags = dict(re.findall(r"#define\s+(RDN_FLAG_\w+)\s+(0x[0-9a-fA-F]+)u", src))
    assert len(flags) == 8, flags
    for name, val in flags.items():
        assert getattr(_abi, name) == int(val, 16), name
    variants = ("RDN_FLAG_DECAYED_RESIDUAL", "RDN_FLAG_PLAIN_COMBINE", "RDN_FLAG_TANH_RESIDUAL",
                "RDN_FLAG_STATELESS_AUX")
    assert _abi.RDN_FLAG_VARIANTS == sum(int(flags[n], 16) for n in variants)


def test_prologue_validation():
    lib = _abi.load()
    a = _abi.PrologueArgs()
    a.rows, a.D, a.dtype, a.eps = 16, 128, _abi.RDN_BF16, 1e-12
    assert lib.rdn_qk_prologue(ctypes.byref(a), None) == 1  # x[0] NULL
    a.x[0], a.y[0] = FAKE, ctypes.c_void_p(0x20000)
    a.D = 96
    assert lib.rdn_qk_prologue(ctypes.byref(a), None) == 2
    a.D = 128
    a.eps = 0.0
    assert lib.rdn_qk_prologue(ctypes.byref(a), None) == 1
    a.eps = 1e-12
    a.y[0] = FAKE  # aliases x
    assert lib.rdn_qk_prologue(ctypes.byref(a), None) == 1
    a.y[0] = ctypes.c_void_p(0x20004)  # misaligned
    assert lib.rdn_qk_prologue(ctypes.byref(a), None) == 6
    a.rows = 0
    assert lib.rdn_qk_prologue_bwd(ctypes.byref(a), None) == 1
    a.rows = 16
    assert lib.rdn_qk_prologue_bwd(ctypes.byref(a), None) == 1  # dy[0] NULL


def test_plain_c_consumer(tmp_path):
    """A C program that includes only include/rdn.h and links librdn.so uses
    the boundary without Python: version, sizes and argument validation (no
    device work, so it runs without a GPU)."""
    _abi.load()
    src = r"""
#include <stdio.h>
#include <string.h>
#include "rdn.h"
int main(void) {
  rdn_fwd_args a;
  memset(&a, 0, sizeof a);
  a.B = 2; a.T = 300; a.H = 4; a.Dk = 128; a.Dv = 128; a.dtype = RDN_BF16;
  a.clip = 1.0f; a.scale = 1.0f;
  size_t ws = 0;
  long long slots = 0;
  if (rdn_fwd_workspace_size(&a, &ws) != RDN_OK || ws == 0) return 1;
  if (rdn_chunk_slots(&a, &slots) != RDN_OK || slots != 2 * 4 * 5) return 2;
  if (rdn_fwd(&a, NULL) != RDN_ERR_INVALID_ARG) return 3;      /* q is NULL */
  if (strstr(rdn_last_error(), "q is NULL") == NULL) return 4;
  a.flags = RDN_FLAG_TANH_RESIDUAL | RDN_FLAG_TIED_GAMMA;
  if (rdn_fwd_workspace_size(&a, &ws) != RDN_OK) return 5;
  a.flags = 0x100u;
  if (rdn_fwd_workspace_size(&a, &ws) != RDN_ERR_UNSUPPORTED) return 6;
  {
    size_t ws2 = 0;  /* the normalised q, k copies: 2 B T H Dk bf16 more */
    a.flags = RDN_FLAG_QK_NORM;
    a.qk_eps = 1e-12f;
    if (rdn_fwd_workspace_size(&a, &ws2) != RDN_OK) return 7;
    a.flags = 0;
    if (rdn_fwd_workspace_size(&a, &ws) != RDN_OK || ws2 != ws + 2u * 2 * 300 * 4 * 128 * 2)
      return 8;
  }
  printf("%s\n", rdn_version());
  return 0;
}
"""
    c = tmp_path / "consumer.c"
    c.write_text(src)
    exe = tmp_path / "consumer"
    libdir = os.path.dirname(_abi.lib_path())
    subprocess.run(["gcc", "-I", os.path.join(ROOT, "include"), str(c), "-o", str(exe),
                    "-L", libdir, "-l:" + os.path.basename(_abi.lib_path()),
                    "-Wl,-rpath," + libdir], check=True)
    r = subprocess.run([str(exe)], capture_output=True, text=True)
    assert r.returncode == 0, (r.returncode, r.stdout, r.stderr)
    assert r.stdout.startswith("rdn-gb300")


@pytest.mark.parametrize("fn", ["rdn_fwd", "rla_fwd", "rdn_bwd", "rla_bwd"])
def test_fault_injection(fn, monkeypatch):
    """RDN_FAULT_INJECT (host side, no GPU needed): a call that passes argument
    validation and the workspace check fails as asked -- "workspace" with
    RDN_ERR_WORKSPACE, "launch" with RDN_ERR_CUDA -- before anything is
    enqueued, and says that the failure was injected."""
    lib = _abi.load()
    ok = dict(q=FAKE, k=FAKE, v=FAKE, g=FAKE, beta=FAKE, gamma=FAKE, o=FAKE)
    n = ctypes.c_size_t(0)
    if fn.endswith("_fwd"):
        a = _fwd_args(**ok)
        assert lib[fn + "_workspace_size"](ctypes.byref(a), ctypes.byref(n)) == 0
    else:
        a = _abi.BwdArgs()
        a.fwd = _fwd_args(**ok)
        for f in ("dO", "dq", "dk", "dv", "dg", "dbeta", "dgamma"):
            setattr(a, f, FAKE)
        assert lib[fn + "_workspace_size"](ctypes.byref(a), ctypes.byref(n)) == 0
    a.workspace, a.workspace_bytes = FAKE, n.value
    for what, status in (("workspace", 5), ("launch", 3)):
        monkeypatch.setenv("RDN_FAULT_INJECT", what)
        assert lib[fn](ctypes.byref(a), None) == status, what
        assert "injected" in lib.rdn_last_error().decode(), what
    # a too-small workspace is still reported as such (validation comes first)
    a.workspace_bytes = n.value - 16
    assert lib[fn](ctypes.byref(a), None) == 5
    assert "injected" not in lib.rdn_last_error().decode()
