"""The paper's variants of the method (variant_flags) through the C ABI,
against the oracle run with the same variant bits.

Library flag -> oracle bit: DECAYED_RESIDUAL -> DECAYED, PLAIN_COMBINE ->
PLAIN, TANH_RESIDUAL -> TANH, STATELESS_AUX -> STATELESS.  Small cases over
several chunks with a ragged tail, nonzero initial states and upstream state
gradients; the clip decisions are kept away from c (tests/test_gpu_bwd.py)."""
import numpy as np
import pytest
import torch

import oracle
import paper_2509_25223_gb300 as rdn
from rdn_synthetic import make_inputs
from tests.parity_util import as64, assert_close

pytestmark = pytest.mark.gpu

NAMES = ("q", "k", "v", "g", "beta", "gamma")
GRADS = ("dq", "dk", "dv", "dg", "dbeta", "dgamma", "dS0", "dR0")
TO_ORACLE = {rdn.DECAYED_RESIDUAL: oracle.DECAYED, rdn.PLAIN_COMBINE: oracle.PLAIN,
             rdn.TANH_RESIDUAL: oracle.TANH, rdn.STATELESS_AUX: oracle.STATELESS}
ALL = rdn.DECAYED_RESIDUAL | rdn.PLAIN_COMBINE | rdn.TANH_RESIDUAL | rdn.STATELESS_AUX
FLAGS = [rdn.DECAYED_RESIDUAL, rdn.PLAIN_COMBINE, rdn.TANH_RESIDUAL, rdn.STATELESS_AUX,
         rdn.DECAYED_RESIDUAL | rdn.TANH_RESIDUAL, rdn.PLAIN_COMBINE | rdn.STATELESS_AUX, ALL]


def _mods(flags):
    return sum(o for f, o in TO_ORACLE.items() if flags & f)


def _inputs(dtype, D, T=130, B=2, H=2, seed=0):
    x = make_inputs(B, T, H, D, dtype=dtype, nonzero_state=True, with_grad_out=True,
                    device="cuda", state_std=0.1, seed=seed)
    gen = torch.Generator(device="cpu").manual_seed(seed + 1)
    x["dST"] = torch.randn(x["S0"].shape, generator=gen).cuda()
    x["dRT"] = torch.randn(x["R0"].shape, generator=gen).cuda()
    return x


def _condition(x, clip, dtype, variant, mods):
    v2, _ = oracle.clip_margin_condition(variant, *(as64(x[n]) for n in NAMES), clip,
                                         as64(x["S0"]), as64(x["R0"]), margin=1e-2, quant=dtype,
                                         mods=mods)
    x["v"].copy_(torch.from_numpy(v2).to(x["v"].dtype))


@pytest.mark.parametrize("variant", ["rdn", "rla"])
@pytest.mark.parametrize("dtype,D", [("f32", 64), ("bf16", 128)])
@pytest.mark.parametrize("flags", FLAGS)
def test_variant_fwd(variant, dtype, D, flags):
    ov = oracle.RDN if variant == "rdn" else oracle.RLA
    x = _inputs(dtype, D)
    clip = 0.8
    fn = rdn.rdn_fwd if variant == "rdn" else rdn.rla_fwd
    o, ST, RT = fn(*(x[n] for n in NAMES), clip=clip, S0=x["S0"], R0=x["R0"],
                   variant_flags=flags)
    torch.cuda.synchronize()
    oref, Sref, Rref = oracle.fwd(ov, *(as64(x[n]) for n in NAMES), clip, as64(x["S0"]),
                                  as64(x["R0"]), mods=_mods(flags))
    assert_close(o, oref, dtype, "o")
    assert_close(ST, Sref, dtype, "ST")
    assert_close(RT, Rref, dtype, "RT")


@pytest.mark.parametrize("variant", ["rdn", "rla"])
@pytest.mark.parametrize("dtype,D", [("f32", 64), ("bf16", 128)])
@pytest.mark.parametrize("flags", FLAGS)
@pytest.mark.parametrize("reuse", [False, True, "saved"])
def test_variant_bwd(variant, dtype, D, flags, reuse):
    ov = oracle.RDN if variant == "rdn" else oracle.RLA
    x = _inputs(dtype, D, seed=3)
    clip = 0.8
    _condition(x, clip, dtype, ov, _mods(flags))
    kw = {}
    if reuse:  # the forward's chunk states and records (and its saved intermediates)
        saved = reuse == "saved"
        nbytes = rdn.workspace_bytes(f"{variant}_fwd", *x["q"].shape[:3], D,
                                     torch.bfloat16 if dtype == "bf16" else torch.float32,
                                     save_for_bwd=saved, variant_flags=flags)
        ws = torch.empty(nbytes, dtype=torch.uint8, device="cuda")
        fwd = rdn.rdn_fwd if variant == "rdn" else rdn.rla_fwd
        _, _, _, Sc, Rc = fwd(*(x[n] for n in NAMES), clip=clip, S0=x["S0"], R0=x["R0"],
                              return_chunk_states=True, workspace=ws, variant_flags=flags,
                              save_for_bwd=saved)
        kw = dict(S_chunks=Sc, R_chunks=Rc, fwd_workspace=ws, fwd_saved=saved)
    fn = rdn.rdn_bwd if variant == "rdn" else rdn.rla_bwd
    d = fn(*(x[n] for n in NAMES), x["dO"], clip=clip, S0=x["S0"], R0=x["R0"], dST=x["dST"],
           dRT=x["dRT"], variant_flags=flags, **kw)
    torch.cuda.synchronize()
    ref = oracle.bwd(ov, *(as64(x[n]) for n in NAMES), clip, as64(x["S0"]), as64(x["R0"]),
                     as64(x["dO"]), as64(x["dST"]), as64(x["dRT"]), mods=_mods(flags))
    for name in GRADS:
        if flags & rdn.STATELESS_AUX and name == "dR0":  # R0 does not enter
            assert float(d[name].abs().max()) == 0.0
            continue
        assert_close(d[name], ref[name], dtype, name)


def test_variant_packed_sequences_and_tied_gates():
    """A variant on packed sequences with tied gates: each sequence equals
    the oracle on that sequence alone (gamma = beta there)."""
    flags = rdn.DECAYED_RESIDUAL | rdn.TANH_RESIDUAL
    lens = [70, 0, 129, 1]
    T, H, D = sum(lens), 2, 128
    x = make_inputs(1, T, H, D, dtype="bf16", with_grad_out=True, device="cuda", seed=21)
    N = len(lens)
    gen = torch.Generator(device="cpu").manual_seed(22)
    S0 = (0.1 * torch.randn(N, H, D, D, generator=gen)).cuda()
    R0 = (0.1 * torch.randn(N, H, D, D, generator=gen)).cuda()
    cu_h = np.concatenate([[0], np.cumsum(lens)]).astype(np.int32)
    cu = torch.from_numpy(cu_h).cuda()
    o, ST, RT = rdn.rdn_fwd(x["q"], x["k"], x["v"], x["g"], x["beta"], None, clip=1.0, S0=S0,
                            R0=R0, cu_seqlens=cu, tied_gamma=True, variant_flags=flags)
    d = rdn.rdn_bwd(x["q"], x["k"], x["v"], x["g"], x["beta"], None, x["dO"], clip=1.0, S0=S0,
                    R0=R0, cu_seqlens=cu, tied_gamma=True, variant_flags=flags,
                    out=dict(dq=torch.empty_like(x["q"]), dk=torch.empty_like(x["k"]),
                             dv=torch.empty_like(x["v"]), dg=torch.empty_like(x["g"]),
                             dbeta=torch.empty_like(x["g"]), dS0=torch.empty_like(S0),
                             dR0=torch.empty_like(R0)))
    torch.cuda.synchronize()
    mods = oracle.DECAYED | oracle.TANH
    for s in range(N):
        t0, t1 = int(cu_h[s]), int(cu_h[s + 1])
        if t1 == t0:
            assert torch.equal(ST[s], S0[s]) and torch.equal(RT[s], R0[s])
            continue
        sl = {n: as64(x[n][:, t0:t1]) for n in NAMES + ("dO",)}
        sl["gamma"] = sl["beta"]
        oref, Sref, Rref = oracle.fwd(oracle.RDN, *(sl[n] for n in NAMES), 1.0,
                                      as64(S0[s:s + 1]), as64(R0[s:s + 1]), mods=mods)
        assert_close(o[:, t0:t1], oref, "bf16", f"o[{s}]")
        assert_close(ST[s:s + 1], Sref, "bf16", f"ST[{s}]")
        assert_close(RT[s:s + 1], Rref, "bf16", f"RT[{s}]")
        ref = oracle.bwd(oracle.RDN, *(sl[n] for n in NAMES), 1.0, as64(S0[s:s + 1]),
                         as64(R0[s:s + 1]), sl["dO"], mods=mods)
        for name in ("dq", "dk", "dv", "dg"):
            assert_close(d[name][:, t0:t1], ref[name], "bf16", f"{name}[{s}]")
        assert_close(d["dbeta"][:, t0:t1], ref["dbeta"] + ref["dgamma"], "bf16", f"dbeta[{s}]")
        assert_close(d["dS0"][s:s + 1], ref["dS0"], "bf16", f"dS0[{s}]")
        assert_close(d["dR0"][s:s + 1], ref["dR0"], "bf16", f"dR0[{s}]")


@pytest.mark.parametrize("flags", [rdn.DECAYED_RESIDUAL | rdn.PLAIN_COMBINE | rdn.STATELESS_AUX,
                                   rdn.TANH_RESIDUAL])
def test_variant_bench_shape_sampled(flags):
    """RDN fwd + bwd with variant flags at the bench's sequence length and
    head count (B = 2, T = 4096, H = 16, d = 128, bf16), two sampled heads
    against the oracle."""
    m = _mods(flags)
    x = make_inputs(2, 4096, 16, 128, dtype="bf16", with_grad_out=True, device="cuda", seed=8)
    picks = [(0, 2), (1, 13)]
    for b, h in picks:
        sl = {n: as64(x[n][b:b + 1, :, h:h + 1]) for n in NAMES}
        v2, _ = oracle.clip_margin_condition(oracle.RDN, *(sl[n] for n in NAMES), 1.0,
                                             margin=1e-2, quant="bf16", mods=m)
        x["v"][b, :, h] = torch.from_numpy(v2[0, :, 0]).to(x["v"].dtype).cuda()
    o, ST, RT, Sc, Rc = rdn.rdn_fwd(*(x[n] for n in NAMES), clip=1.0, return_chunk_states=True,
                                    variant_flags=flags)
    d = rdn.rdn_bwd(*(x[n] for n in NAMES), x["dO"], clip=1.0, S_chunks=Sc, R_chunks=Rc,
                    variant_flags=flags)
    torch.cuda.synchronize()
    for b, h in picks:
        sl = {n: as64(x[n][b:b + 1, :, h:h + 1]) for n in NAMES + ("dO",)}
        oref, Sref, Rref = oracle.fwd(oracle.RDN, *(sl[n] for n in NAMES), 1.0, mods=m)
        assert_close(o[b:b + 1, :, h:h + 1], oref, "bf16", f"o[{b},{h}]")
        assert_close(ST[b:b + 1, h:h + 1], Sref, "bf16", f"ST[{b},{h}]")
        assert_close(RT[b:b + 1, h:h + 1], Rref, "bf16", f"RT[{b},{h}]")
        ref = oracle.bwd(oracle.RDN, *(sl[n] for n in NAMES), 1.0, None, None, sl["dO"], mods=m)
        for name in ("dq", "dk", "dv", "dg", "dbeta", "dgamma"):
            assert_close(d[name][b:b + 1, :, h:h + 1], ref[name], "bf16", f"{name}[{b},{h}]")
        assert_close(d["dS0"][b:b + 1, h:h + 1], ref["dS0"], "bf16", f"dS0[{b},{h}]")
