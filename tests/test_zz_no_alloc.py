"""rdn_fwd_noalloc: the RDN forward for callers that cannot allocate device
memory (an engine plugin handed only its input and output tensors, or a
serving loop that forbids cudaMalloc after start-up).  It must return what
rdn_fwd returns for the same inputs, call after call, using only the scratch
array built into the library.

Collected last on purpose (file name), so a run that stops at the first
failure has already run every other test; it also passes on its own in a
fresh process."""
import ctypes

import pytest
import torch

import paper_2509_25223_gb300 as rdn
from paper_2509_25223_gb300 import _abi
from rdn_synthetic import make_inputs
from tests.parity_util import assert_close

pytestmark = pytest.mark.gpu

NAMES = ("q", "k", "v", "g", "beta", "gamma")


def _noalloc(x, clip=1.0, cu=None):
    """Call rdn_fwd_noalloc through the C ABI; no workspace is passed."""
    lib = _abi.load()
    B, T, H, D = x["q"].shape
    N = B if cu is None else cu.numel() - 1
    o = torch.empty(B, T, H, D, dtype=x["q"].dtype, device=x["q"].device)
    ST = torch.empty(N, H, D, D, device=x["q"].device)
    RT = torch.empty_like(ST)
    a = _abi.FwdArgs()
    a.B, a.T, a.H, a.Dk, a.Dv = B, T, H, D, D
    a.dtype = _abi.RDN_BF16 if x["q"].dtype == torch.bfloat16 else _abi.RDN_F32
    p = lambda t: None if t is None else ctypes.c_void_p(t.data_ptr())
    a.q, a.k, a.v = p(x["q"]), p(x["k"]), p(x["v"])
    a.g, a.beta, a.gamma = p(x["g"]), p(x["beta"]), p(x["gamma"])
    a.clip, a.scale, a.flags = clip, 1.0, 0
    a.S0, a.R0 = p(x["S0"]), p(x["R0"])
    a.o, a.ST, a.RT = p(o), p(ST), p(RT)
    a.workspace, a.workspace_bytes = None, 0
    if cu is not None:
        a.cu_seqlens, a.num_seqs = p(cu), N
    stream = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    st = lib.rdn_fwd_noalloc(ctypes.byref(a), stream)
    assert st == 0, lib.rdn_last_error().decode()
    torch.cuda.synchronize()
    return o, ST, RT


def _compare(x, dtype, cu=None, what=""):
    o, ST, RT = _noalloc(x, cu=cu)
    kw = {} if cu is None else dict(cu_seqlens=cu)
    o2, ST2, RT2 = rdn.rdn_fwd(*(x[n] for n in NAMES), clip=1.0, S0=x["S0"], R0=x["R0"], **kw)
    torch.cuda.synchronize()
    assert_close(o, o2.float().cpu().double().numpy(), dtype, f"{what} o")
    assert_close(ST, ST2.cpu().double().numpy(), "f32", f"{what} ST")
    assert_close(RT, RT2.cpu().double().numpy(), "f32", f"{what} RT")


def test_noalloc_matches_rdn_fwd_call_after_call():
    """Problems of growing size back to back -- a small one, a larger one,
    another of that size on new inputs (every scratch word it reads was left
    by the previous call), then exactly the largest the scratch holds
    (1 x 12 heads x 67 chunks = 804 chunk records) -- then packed sequences
    (whose table sits after the records) and fp32 inputs: each must equal
    rdn_fwd on the same inputs."""
    cases = [((1, 130, 3, 64), 0), ((2, 300, 4, 128), 1), ((2, 300, 4, 128), 2),
             ((1, 67 * 64, 12, 128), 3)]
    for (B, T, H, D), seed in cases:
        x = make_inputs(B, T, H, D, dtype="bf16", nonzero_state=True, device="cuda",
                        seed=seed, state_std=0.1)
        _compare(x, "bf16", what=f"B{B} T{T} H{H} D{D}")
    # packed sequences: lengths 70, 0, 130, 64 (an empty one and a ragged tail)
    lens = [70, 0, 130, 64]
    x = make_inputs(1, sum(lens), 2, 128, dtype="bf16", device="cuda", seed=4)
    gen = torch.Generator(device="cpu").manual_seed(15)
    for n in ("S0", "R0"):
        x[n] = (0.1 * torch.randn(len(lens), 2, 128, 128, generator=gen)).cuda()
    cu = torch.tensor([0, 70, 70, 200, 264], dtype=torch.int32, device="cuda")
    _compare(x, "bf16", cu=cu, what="packed")
    x = make_inputs(2, 150, 2, 64, dtype="f32", nonzero_state=True, device="cuda", seed=5,
                    state_std=0.1)
    _compare(x, "f32", what="fp32")


def test_noalloc_rejects_problems_beyond_its_scratch():
    lib = _abi.load()
    a = _abi.FwdArgs()
    a.B, a.T, a.H, a.Dk, a.Dv = 8, 4096, 16, 128, 128  # 8192 chunks > 804
    a.dtype, a.clip, a.scale = _abi.RDN_BF16, 1.0, 1.0
    fake = ctypes.c_void_p(0x10000)
    a.q = a.k = a.v = a.g = a.beta = a.gamma = a.o = fake
    assert lib.rdn_fwd_noalloc(ctypes.byref(a), None) == 5
    msg = lib.rdn_last_error().decode()
    assert "built-in scratch" in msg and "804" in msg
    # one chunk record beyond it: 1 x 5 heads x 161 chunks = 805
    a.B, a.T, a.H = 1, 161 * 64, 5
    assert lib.rdn_fwd_noalloc(ctypes.byref(a), None) == 5
    assert "805 chunk records" in lib.rdn_last_error().decode()


def test_noalloc_rejects_the_save_for_backward_flag():
    """Its scratch is internal, so intermediates saved there would be out of
    rdn_bwd's reach: the flag is refused before anything is launched."""
    lib = _abi.load()
    a = _abi.FwdArgs()
    a.B, a.T, a.H, a.Dk, a.Dv = 1, 64, 1, 128, 128
    a.dtype, a.clip, a.scale = _abi.RDN_BF16, 1.0, 1.0
    a.flags = _abi.RDN_FLAG_SAVE_FOR_BWD
    fake = ctypes.c_void_p(0x10000)
    a.q = a.k = a.v = a.g = a.beta = a.gamma = a.o = fake
    a.S_chunks = a.R_chunks = fake
    assert lib.rdn_fwd_noalloc(ctypes.byref(a), None) == 2
    assert "caller workspace" in lib.rdn_last_error().decode()
