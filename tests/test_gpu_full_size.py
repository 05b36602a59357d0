"""Full-size parity: every (b, h) head of the bf16 workloads against the fp64
oracle, through the C ABI, in the launch configuration bench.py times.

  rdn_fwd_bf16_B8H16T2048D128           forward, zero states
  rdn_fwd_bf16_B2H16T16384D128_state    forward, S0, R0 ~ N(0, 0.02^2), final states
  rdn_fwd_bwd_bf16_B8H16T4096D128       forward (chunk states, saved
                                        intermediates) + backward, dO ~ N(0, 1)

each for RDN and for RLA.  The oracle runs all heads at once (OpenMP over
(b, h)).  The bound is max |gpu - ref| <= 2e-2 RMS(ref) per tensor; tensors the
library returns in fp32 (final states, gate gradients, dS0, dR0) are held to it
as stated, bf16-typed ones (o, dq, dk, dv) may add half a bf16 ulp of their own
store rounding (tests/parity_util.py).  Each workload also runs with
RDN_FLAG_F32_OUT (the same computation, o, dq, dk, dv returned in fp32), and
there every tensor is held to the plain bound.  With RDN_PARITY_REPORT=<file> every
compared tensor appends its statistics (plain max|err|/RMS, RMS error / RMS,
elements beyond the plain bound) to that file."""
import numpy as np
import pytest
import torch

import oracle
import paper_2509_25223_gb300 as rdn
from rdn_synthetic import WORKLOADS, make_workload_inputs
from tests.parity_util import as64, assert_close, record

pytestmark = pytest.mark.gpu

NAMES = ("q", "k", "v", "g", "beta", "gamma")
GRADS = ("dq", "dk", "dv", "dg", "dbeta", "dgamma", "dS0", "dR0")
MARGIN = 1e-2  # the clip-margin conditioner's margin (as in tests/test_gpu_bwd.py)


def _check(test, name, gpu, ref, **extra):
    s = record(test, name, gpu, ref, **extra)
    assert_close(gpu, ref, "bf16", f"{test}: {name}")
    return s


@pytest.mark.parametrize("variant", ["rdn", "rla"])
@pytest.mark.parametrize("wname", ["rdn_fwd_bf16_B8H16T2048D128",
                                   "rdn_fwd_bf16_B2H16T16384D128_state"])
def test_fwd_full_size_all_heads(variant, wname):
    w = WORKLOADS[wname]
    x = make_workload_inputs(w, device="cuda")
    fn = rdn.rdn_fwd if variant == "rdn" else rdn.rla_fwd
    o, ST, RT = fn(*(x[n] for n in NAMES), clip=w.clip, S0=x["S0"], R0=x["R0"])
    o32, _, _ = fn(*(x[n] for n in NAMES), clip=w.clip, S0=x["S0"], R0=x["R0"], f32_out=True)
    torch.cuda.synchronize()
    assert o32.dtype == torch.float32 and torch.equal(o32.to(torch.bfloat16), o)
    v = oracle.RDN if variant == "rdn" else oracle.RLA
    oref, Sref, Rref = oracle.fwd(v, *(as64(x[n]) for n in NAMES), w.clip, as64(x["S0"]),
                                  as64(x["R0"]))
    test = f"{variant} fwd {wname}"
    _check(test, "o", o, oref)
    _check(test, "o (fp32 out)", o32, oref)
    _check(test, "ST", ST, Sref)
    _check(test, "RT", RT, Rref)


@pytest.mark.parametrize("variant", ["rdn", "rla"])
def test_fwd_bwd_full_size_all_heads(variant):
    """The bench step's workload and options, all 128 heads.  The inputs are
    first conditioned so that every fp64 clip decision has a margin (the
    count of moved v elements is recorded)."""
    w = WORKLOADS["rdn_fwd_bwd_bf16_B8H16T4096D128"]
    x = make_workload_inputs(w, device="cuda")
    v = oracle.RDN if variant == "rdn" else oracle.RLA
    a = {n: as64(x[n]) for n in NAMES}
    v2, moved = oracle.clip_margin_condition(v, a["q"], a["k"], a["v"], a["g"], a["beta"],
                                             a["gamma"], w.clip, None, None, margin=MARGIN,
                                             quant="bf16")
    x["v"] = torch.from_numpy(v2).to(torch.bfloat16).cuda()
    a["v"] = as64(x["v"])
    wsf = torch.empty(rdn.workspace_bytes(f"{variant}_fwd", w.B, w.T, w.H, w.D,
                                          save_for_bwd=True), dtype=torch.uint8, device="cuda")
    fwd = rdn.rdn_fwd if variant == "rdn" else rdn.rla_fwd
    bwd = rdn.rdn_bwd if variant == "rdn" else rdn.rla_bwd
    o, ST, RT, Sc, Rc = fwd(*(x[n] for n in NAMES), clip=w.clip, return_chunk_states=True,
                            workspace=wsf, save_for_bwd=True)
    d = bwd(*(x[n] for n in NAMES), x["dO"], clip=w.clip, S_chunks=Sc, R_chunks=Rc,
            fwd_workspace=wsf, fwd_saved=True)
    # the same step with fp32 results
    o32, _, _, Sc2, Rc2 = fwd(*(x[n] for n in NAMES), clip=w.clip, return_chunk_states=True,
                              workspace=wsf, save_for_bwd=True, f32_out=True)
    d32 = bwd(*(x[n] for n in NAMES), x["dO"], clip=w.clip, S_chunks=Sc2, R_chunks=Rc2,
              fwd_workspace=wsf, fwd_saved=True, f32_out=True)
    torch.cuda.synchronize()
    assert torch.equal(o32.to(torch.bfloat16), o)
    for name in ("dq", "dk", "dv"):
        assert d32[name].dtype == torch.float32
        assert torch.equal(d32[name].to(torch.bfloat16), d[name]), name
    ref = oracle.bwd(v, *(a[n] for n in NAMES), w.clip, None, None, as64(x["dO"]))
    oref, Sref, Rref = oracle.fwd(v, *(a[n] for n in NAMES), w.clip, None, None)
    test = f"{variant} fwd+bwd {w.name}"
    extra = dict(conditioner_moved=moved, conditioner_margin=MARGIN)
    _check(test, "o", o, oref, **extra)
    _check(test, "ST", ST, Sref, **extra)
    _check(test, "RT", RT, Rref, **extra)
    _check(test, "o (fp32 out)", o32, oref, **extra)
    for name in GRADS:
        assert torch.isfinite(d[name].float()).all(), name
        _check(test, name, d[name], ref[name], **extra)
    for name in ("dq", "dk", "dv"):
        _check(test, f"{name} (fp32 out)", d32[name], ref[name], **extra)


@pytest.mark.parametrize("mode", ["tanh_residual", "stateless_aux", "qk_norm"])
def test_fwd_bwd_full_size_modes(mode):
    """The bench step (RDN, all 128 heads, the step's options) with one of
    the tensor-core modes beyond the method: the tanh residual and the
    stateless correction (variant flags, the oracle's mods bits), or the q, k
    normalisation inside the library (q, k taken as raw x; the reference is
    the oracle's prologue, rounded to bf16 as the library holds it, then its
    recurrence, and dq, dk through the prologue's backward at x)."""
    w = WORKLOADS["rdn_fwd_bwd_bf16_B8H16T4096D128"]
    x = make_workload_inputs(w, device="cuda")
    flags = {"tanh_residual": rdn.TANH_RESIDUAL, "stateless_aux": rdn.STATELESS_AUX}.get(mode, 0)
    mods = {"tanh_residual": oracle.TANH, "stateless_aux": oracle.STATELESS}.get(mode, 0)
    qkn = mode == "qk_norm"
    if qkn:  # raw x moved off the bf16 rounding ties of y (tests/test_gpu_qk_norm.py)
        for n in ("q", "k"):
            xc, _ = oracle.qk_round_margin_condition(as64(x[n]), 1e-12)
            x[n] = torch.from_numpy(xc).to(torch.bfloat16).cuda()
    a = {n: as64(x[n]) for n in NAMES}
    if qkn:
        for n in ("q", "k"):
            y = oracle.qk_prologue(a[n], 1e-12)
            a[n] = as64(torch.from_numpy(y).to(torch.bfloat16))
    v2, moved = oracle.clip_margin_condition(oracle.RDN, a["q"], a["k"], a["v"], a["g"],
                                             a["beta"], a["gamma"], w.clip, None, None,
                                             margin=MARGIN, quant="bf16", mods=mods)
    x["v"] = torch.from_numpy(v2).to(torch.bfloat16).cuda()
    a["v"] = as64(x["v"])
    wsf = torch.empty(rdn.workspace_bytes("rdn_fwd", w.B, w.T, w.H, w.D, save_for_bwd=True,
                                          variant_flags=flags, qk_norm=qkn),
                      dtype=torch.uint8, device="cuda")
    kw = dict(clip=w.clip, variant_flags=flags, qk_norm=qkn)
    o, ST, RT, Sc, Rc = rdn.rdn_fwd(*(x[n] for n in NAMES), return_chunk_states=True,
                                    workspace=wsf, save_for_bwd=True, **kw)
    d = rdn.rdn_bwd(*(x[n] for n in NAMES), x["dO"], S_chunks=Sc, R_chunks=Rc,
                    fwd_workspace=wsf, fwd_saved=True, **kw)
    torch.cuda.synchronize()
    assert rdn.device_status() == 0
    oref, Sref, Rref = oracle.fwd(oracle.RDN, *(a[n] for n in NAMES), w.clip, None, None,
                                  mods=mods)
    ref = oracle.bwd(oracle.RDN, *(a[n] for n in NAMES), w.clip, None, None, as64(x["dO"]),
                     mods=mods)
    if qkn:
        ref["dq"] = oracle.qk_prologue_bwd(as64(x["q"]), ref["dq"], 1e-12)
        ref["dk"] = oracle.qk_prologue_bwd(as64(x["k"]), ref["dk"], 1e-12)
    test = f"rdn fwd+bwd {w.name} {mode}"
    extra = dict(conditioner_moved=moved, conditioner_margin=MARGIN)
    _check(test, "o", o, oref, **extra)
    _check(test, "ST", ST, Sref, **extra)
    _check(test, "RT", RT, Rref, **extra)
    for name in GRADS:
        assert torch.isfinite(d[name].float()).all(), name
        if mode == "stateless_aux" and name == "dR0":
            assert float(d[name].abs().max()) == 0.0  # R0 enters nothing
            continue
        _check(test, name, d[name], ref[name], **extra)
