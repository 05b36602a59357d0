"""RDN_FLAG_QK_NORM: the q/k activation and normalisation applied inside the
library, y = SiLU(x) / max(||SiLU(x)||, eps) per row, against the oracle's
chain prologue -> recurrence (and, backwards, recurrence -> prologue).

q and k are raw projections x (normal draws, not normalised).  The library
holds y in the input dtype (as a caller's own prologue pass would), so the
reference rounds the oracle's fp64 y to that dtype before the recurrence,
exactly as the other tests hand the oracle the bf16 q, k the kernels read;
the backward's Jacobian is the oracle's, at the fp64 x.  The rounding of y
to bf16 is a decision the two sides take in different precisions (fp32 in
the library, fp64 in the oracle), so the raw rows are first conditioned
(oracle.qk_round_margin_condition: x moved by bf16 steps) until every fp64 y
is a margin away from a bf16 rounding tie; both then hold the same y.  The
clip mask is made unique the usual way (v moved until every fp64 residual is
a margin away from c), on the y the reference uses."""
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
EPS = 1e-12
MARGIN = 1e-2


def _inputs(B, T, H, D, dtype, seed=0, zero_row=False):
    x = make_inputs(B, T, H, D, dtype=dtype, nonzero_state=True, with_grad_out=True,
                    device="cuda", state_std=0.1, seed=seed)
    gen = torch.Generator(device="cpu").manual_seed(seed + 100)
    td = x["q"].dtype
    for n in ("q", "k"):  # raw projections, conditioned (bf16 y: see the module's text)
        raw = torch.randn(B, T, H, D, generator=gen).to(td)
        if td == torch.bfloat16:
            raw = torch.from_numpy(oracle.qk_round_margin_condition(raw, EPS)[0]).to(td)
        x[n] = raw.cuda()
    if zero_row:  # a row whose norm is below eps: y = u / eps = 0, du = dy / eps
        x["k"][0, 0, 0] = 0
        x["q"][0, T - 1, H - 1] = 0
    return x


def _oracle_y(x):
    """The oracle's y, rounded to the dtype the library holds it in."""
    td = x["q"].dtype
    rnd = lambda y: as64(torch.from_numpy(y).to(td))  # noqa: E731
    return (rnd(oracle.qk_prologue(as64(x["q"]), EPS)),
            rnd(oracle.qk_prologue(as64(x["k"]), EPS)))


def _condition(x, clip, dtype, variant):
    yq, yk = _oracle_y(x)
    v2, _ = oracle.clip_margin_condition(variant, yq, yk, as64(x["v"]), as64(x["g"]),
                                         as64(x["beta"]), as64(x["gamma"]), clip,
                                         as64(x["S0"]), as64(x["R0"]), margin=MARGIN,
                                         quant=dtype)
    x["v"] = torch.from_numpy(v2).to(x["v"].dtype).cuda()


def _ref_fwd(x, clip, variant):
    yq, yk = _oracle_y(x)
    return oracle.fwd(variant, yq, yk, *(as64(x[n]) for n in NAMES[2:]), clip,
                      as64(x["S0"]), as64(x["R0"]))


def _ref_bwd(x, clip, variant, dST, dRT):
    yq, yk = _oracle_y(x)
    d = oracle.bwd(variant, yq, yk, *(as64(x[n]) for n in NAMES[2:]), clip, as64(x["S0"]),
                   as64(x["R0"]), as64(x["dO"]), as64(dST), as64(dRT))
    d["dq"] = oracle.qk_prologue_bwd(as64(x["q"]), d["dq"], EPS)
    d["dk"] = oracle.qk_prologue_bwd(as64(x["k"]), d["dk"], EPS)
    return d


def _fns(variant):
    return (rdn.rdn_fwd, rdn.rdn_bwd) if variant == oracle.RDN else (rdn.rla_fwd, rdn.rla_bwd)


# bf16 with D = 128 runs the tensor-core kernels (normalisation fused into the
# per-chunk pass; the backward's gradients w.r.t. y kept in fp32 for one
# Jacobian pass); the others the prologue kernels around the fp32 chunk kernels
CASES = [("bf16", 128), ("bf16", 64), ("f32", 128), ("f32", 64)]


@pytest.mark.parametrize("variant", [oracle.RDN, oracle.RLA])
@pytest.mark.parametrize("dtype,D", CASES)
def test_qk_norm_fwd_bwd(variant, dtype, D):
    clip = 1.0
    x = _inputs(2, 130, 2, D, dtype)
    _condition(x, clip, dtype, variant)
    fwd, bwd = _fns(variant)
    o, ST, RT = fwd(*(x[n] for n in NAMES), clip=clip, S0=x["S0"], R0=x["R0"], qk_norm=True,
                    qk_eps=EPS)
    ro, rST, rRT = _ref_fwd(x, clip, variant)
    assert_close(o, ro, dtype, "o")
    assert_close(ST, rST, dtype, "ST")
    assert_close(RT, rRT, dtype, "RT")
    gen = torch.Generator(device="cpu").manual_seed(5)
    dST = torch.randn(x["S0"].shape, generator=gen).cuda()
    dRT = torch.randn(x["R0"].shape, generator=gen).cuda()
    d = bwd(*(x[n] for n in NAMES), x["dO"], clip=clip, S0=x["S0"], R0=x["R0"], dST=dST,
            dRT=dRT, qk_norm=True, qk_eps=EPS)
    torch.cuda.synchronize()
    ref = _ref_bwd(x, clip, variant, dST, dRT)
    for name in GRADS:
        assert_close(d[name], ref[name], dtype, name)
    assert rdn.device_status() == 0


@pytest.mark.parametrize("dtype,D", [("bf16", 128), ("f32", 64)])
def test_qk_norm_floored_rows(dtype, D):
    """Rows whose ||SiLU(x)|| is below eps (here x = 0): y = u / eps = 0 and
    dy / eps passes back, a gain of 1 / eps.  Those rows and the others are
    each held to the bound relative to their own RMS."""
    clip = 1.0
    x = _inputs(2, 130, 2, D, dtype, seed=2, zero_row=True)
    _condition(x, clip, dtype, oracle.RDN)
    o, _, _ = rdn.rdn_fwd(*(x[n] for n in NAMES), clip=clip, S0=x["S0"], R0=x["R0"],
                          qk_norm=True, qk_eps=EPS)
    d = rdn.rdn_bwd(*(x[n] for n in NAMES), x["dO"], clip=clip, S0=x["S0"], R0=x["R0"],
                    qk_norm=True, qk_eps=EPS)
    torch.cuda.synchronize()
    assert_close(o, _ref_fwd(x, clip, oracle.RDN)[0], dtype, "o")
    ref = _ref_bwd(x, clip, oracle.RDN, None, None)
    for name, (b, t, h) in (("dk", (0, 0, 0)), ("dq", (0, 129, 1))):
        g, r = d[name], ref[name]
        floored = torch.zeros(g.shape[:3], dtype=torch.bool)
        floored[b, t, h] = True
        m = floored.numpy()
        assert np.abs(r[m]).max() > 1e6  # the 1 / eps gain, taken out before comparing
        assert_close(g[floored.cuda()].double() * EPS, r[m] * EPS, dtype, name + " floored")
        assert_close(g[~floored.cuda()], r[~m], dtype, name + " others")


@pytest.mark.parametrize("variant", [oracle.RDN, oracle.RLA])
def test_qk_norm_saved_forward(variant):
    """The backward reading the forward's workspace (its records, saved
    intermediates and normalised q, k), the one given only the chunk states
    and the one that recomputes everything agree, and all match the oracle."""
    clip = 1.0
    x = _inputs(2, 200, 2, 128, "bf16", seed=3)
    _condition(x, clip, "bf16", variant)
    fwd, bwd = _fns(variant)
    ws = torch.empty(rdn.workspace_bytes("rdn_fwd" if variant == oracle.RDN else "rla_fwd",
                                         2, 200, 2, 128, save_for_bwd=True, qk_norm=True),
                     dtype=torch.uint8, device="cuda")
    o, ST, RT, Sc, Rc = fwd(*(x[n] for n in NAMES), clip=clip, S0=x["S0"], R0=x["R0"],
                            return_chunk_states=True, workspace=ws, save_for_bwd=True,
                            qk_norm=True, qk_eps=EPS)
    kw = dict(clip=clip, S0=x["S0"], R0=x["R0"], qk_norm=True, qk_eps=EPS)
    d_saved = bwd(*(x[n] for n in NAMES), x["dO"], S_chunks=Sc, R_chunks=Rc, fwd_workspace=ws,
                  fwd_saved=True, **kw)
    d_states = bwd(*(x[n] for n in NAMES), x["dO"], S_chunks=Sc, R_chunks=Rc, **kw)
    d_full = bwd(*(x[n] for n in NAMES), x["dO"], **kw)
    torch.cuda.synchronize()
    ref = _ref_bwd(x, clip, variant, None, None)
    for name in GRADS:  # (the saved E, E2 and the recomputed ones round alike up to fp32 order)
        torch.testing.assert_close(d_saved[name].float(), d_full[name].float(), atol=1e-5,
                                   rtol=8e-3)
        torch.testing.assert_close(d_states[name].float(), d_full[name].float(), atol=1e-5,
                                   rtol=8e-3)
        for d in (d_saved, d_states, d_full):
            assert_close(d[name], ref[name], "bf16", name)


def test_qk_norm_matches_separate_prologue():
    """The fused normalisation and the standalone prologue kernel followed by
    the plain forward agree to within a bf16 ulp of y (the two sum the
    squares in different orders)."""
    x = _inputs(2, 150, 2, 128, "bf16", seed=9)
    _condition(x, 1.0, "bf16", oracle.RDN)
    o1, _, _ = rdn.rdn_fwd(*(x[n] for n in NAMES), clip=1.0, S0=x["S0"], R0=x["R0"],
                           qk_norm=True, qk_eps=EPS)
    yq, yk = rdn.qk_prologue(x["q"], x["k"], eps=EPS)
    xs = dict(x, q=yq, k=yk)
    o2, _, _ = rdn.rdn_fwd(*(xs[n] for n in NAMES), clip=1.0, S0=x["S0"], R0=x["R0"])
    torch.cuda.synchronize()
    ro, _, _ = _ref_fwd(x, 1.0, oracle.RDN)
    assert_close(o1, ro, "bf16", "o fused")
    assert_close(o2, ro, "bf16", "o separate")
    rms = float(np.sqrt(np.mean(as64(o2) ** 2)))
    assert float(np.abs(as64(o1) - as64(o2)).max()) <= 2e-2 * rms


def test_qk_norm_packed_sequences():
    """cu_seqlens with the flag: each sequence as its own call."""
    clip = 1.0
    lens = [70, 0, 130, 64]
    T = sum(lens)
    x = _inputs(1, T, 2, 128, "bf16", seed=4)
    x["S0"] = x["R0"] = None
    _condition(x, clip, "bf16", oracle.RDN)
    cu = torch.tensor(np.cumsum([0] + lens), dtype=torch.int32, device="cuda")
    o, ST, RT = rdn.rdn_fwd(*(x[n] for n in NAMES), clip=clip, cu_seqlens=cu, qk_norm=True,
                            qk_eps=EPS)
    d = rdn.rdn_bwd(*(x[n] for n in NAMES), x["dO"], clip=clip, cu_seqlens=cu, qk_norm=True,
                    qk_eps=EPS)
    torch.cuda.synchronize()
    t0 = 0
    for s, L in enumerate(lens):
        if L == 0:
            continue
        sl = {n: x[n][:, t0:t0 + L] for n in NAMES + ("dO",)}
        sl.update(S0=None, R0=None)
        ro, rST, _ = _ref_fwd(sl, clip, oracle.RDN)
        assert_close(o[:, t0:t0 + L], ro, "bf16", f"o[{s}]")
        assert_close(ST[s:s + 1], rST, "bf16", f"ST[{s}]")
        ref = _ref_bwd(sl, clip, oracle.RDN, None, None)
        for name in ("dq", "dk", "dv", "dg"):
            assert_close(d[name][:, t0:t0 + L], ref[name], "bf16", f"{name}[{s}]")
        t0 += L


def test_qk_norm_f32_out():
    """fp32 results with the flag: the plain bound holds."""
    clip = 1.0
    x = _inputs(2, 130, 2, 128, "bf16", seed=6)
    _condition(x, clip, "bf16", oracle.RDN)
    o, _, _ = rdn.rdn_fwd(*(x[n] for n in NAMES), clip=clip, S0=x["S0"], R0=x["R0"],
                          qk_norm=True, qk_eps=EPS, f32_out=True)
    d = rdn.rdn_bwd(*(x[n] for n in NAMES), x["dO"], clip=clip, S0=x["S0"], R0=x["R0"],
                    qk_norm=True, qk_eps=EPS, f32_out=True)
    torch.cuda.synchronize()
    assert o.dtype == torch.float32 and d["dq"].dtype == torch.float32
    assert_close(o, _ref_fwd(x, clip, oracle.RDN)[0], "bf16", "o")
    ref = _ref_bwd(x, clip, oracle.RDN, None, None)
    for name in ("dq", "dk", "dv"):
        assert_close(d[name], ref[name], "bf16", name)


@pytest.mark.parametrize("variant", ["rdn", "rla"])
@pytest.mark.parametrize("dtype,D", [("bf16", 128), ("f32", 64)])
def test_qk_norm_decode_step(variant, dtype, D):
    """rdn_decode_step with the flag: one token, normalised in the step."""
    N, H = 3, 2
    gen = torch.Generator(device="cpu").manual_seed(21)
    td = torch.bfloat16 if dtype == "bf16" else torch.float32
    q = torch.randn(N, H, D, generator=gen).to(td).cuda()
    k = torch.randn(N, H, D, generator=gen).to(td).cuda()
    v = torch.randn(N, H, D, generator=gen).to(td).cuda()
    g = -torch.rand(N, H, generator=gen).cuda()
    beta = torch.rand(N, H, generator=gen).cuda()
    gamma = torch.rand(N, H, generator=gen).cuda()
    S = (0.1 * torch.randn(N, H, D, D, generator=gen)).cuda()
    R = (0.1 * torch.randn(N, H, D, D, generator=gen)).cuda()
    S0, R0 = S.clone(), R.clone()
    o = rdn.rdn_decode_step(q, k, v, g, beta, gamma, S, R, clip=1.0, variant=variant,
                            qk_norm=True, qk_eps=EPS)
    torch.cuda.synchronize()
    yq, yk = _oracle_y({"q": q, "k": k})
    ov = oracle.RDN if variant == "rdn" else oracle.RLA
    ro, rS, rR = oracle.decode_step(ov, yq, yk, as64(v), as64(g), as64(beta), as64(gamma), 1.0,
                                    as64(S0), as64(R0))
    assert_close(o, ro, dtype, "o")
    assert_close(S, rS, dtype, "S")
    assert_close(R, rR, dtype, "R")


def test_qk_norm_decode_chain_equals_forward():
    """T decode steps with the flag give the forward's o and final states."""
    B, T, H, D = 2, 70, 2, 128
    x = _inputs(B, T, H, D, "bf16", seed=8)
    _condition(x, 1.0, "bf16", oracle.RDN)
    o, ST, RT = rdn.rdn_fwd(*(x[n] for n in NAMES), clip=1.0, S0=x["S0"], R0=x["R0"],
                            qk_norm=True, qk_eps=EPS)
    S, R = x["S0"].clone(), x["R0"].clone()
    od = torch.empty_like(o)
    for t in range(T):
        od[:, t] = rdn.rdn_decode_step(*(x[n][:, t].contiguous() for n in NAMES), S, R,
                                       clip=1.0, qk_norm=True, qk_eps=EPS)
    torch.cuda.synchronize()
    ro, rST, rRT = _ref_fwd(x, 1.0, oracle.RDN)
    assert_close(od, ro, "bf16", "o (decode)")
    assert_close(o, ro, "bf16", "o (forward)")
    assert_close(S, rST, "bf16", "S (decode)")
    assert_close(R, rRT, "bf16", "R (decode)")
