"""Parity of rdn_bwd with the oracle's back-propagation through time.

The derivative of the clip jumps at |v - S_{t-1}k| = c, so before each
comparison the inputs are conditioned with the oracle (v moved, in steps
representable in the input dtype, until every fp64 residual is at least a
margin away from c).  The clip mask is then unique at tolerance level and so
is the gradient; see oracle.clip_margin_condition."""
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
MARGIN = 1e-2


def _condition(x, clip, dtype, heads=None, variant=oracle.RDN):
    """Move v (in place on the device tensor) so the fp64 clip decisions have
    a margin; only the listed (b, h) heads when given."""
    sel = heads if heads is not None else [(b, h) for b in range(x["q"].shape[0])
                                           for h in range(x["q"].shape[2])]
    for b, h in sel:
        sl = {n: as64(x[n][b:b + 1, :, h:h + 1]) for n in NAMES}
        S0 = None if x["S0"] is None else as64(x["S0"][b:b + 1, h:h + 1])
        R0 = None if x["R0"] is None else as64(x["R0"][b:b + 1, h:h + 1])
        v2, _ = oracle.clip_margin_condition(variant, sl["q"], sl["k"], sl["v"], sl["g"],
                                             sl["beta"], sl["gamma"], clip, S0, R0,
                                             margin=MARGIN, quant=dtype)
        x["v"][b, :, h] = torch.from_numpy(v2[0, :, 0]).to(x["v"].dtype).to(x["v"].device)


def _ref(x, clip, dST=None, dRT=None, heads=None, scale=1.0, variant=oracle.RDN):
    if heads is None:
        return oracle.bwd(variant, *(as64(x[n]) for n in NAMES), clip, as64(x["S0"]),
                          as64(x["R0"]), as64(x["dO"]), as64(dST), as64(dRT), scale=scale)
    outs = []
    for b, h in heads:
        sl = lambda t: None if t is None else as64(t[b:b + 1, :, h:h + 1])
        st = lambda t: None if t is None else as64(t[b:b + 1, h:h + 1])
        outs.append(oracle.bwd(variant, *(sl(x[n]) for n in NAMES), clip, st(x["S0"]),
                               st(x["R0"]), sl(x["dO"]), st(dST), st(dRT)))
    return outs


def _gpu(x, clip, dST=None, dRT=None, variant="rdn", **kw):
    fn = rdn.rdn_bwd if variant == "rdn" else rdn.rla_bwd
    d = fn(*(x[n] for n in NAMES), x["dO"], clip=clip, S0=x["S0"], R0=x["R0"], dST=dST, dRT=dRT,
           **kw)
    torch.cuda.synchronize()
    return d


@pytest.mark.parametrize("dtype", ["bf16", "f32"])
@pytest.mark.parametrize("D", [64, 128])
@pytest.mark.parametrize("T", [1, 2, 7, 8, 63, 64, 65, 200])
def test_bwd_small(dtype, D, T):
    clip = 1.0
    x = make_inputs(2, T, 2, D, dtype=dtype, nonzero_state=True, with_grad_out=True,
                    device="cuda", state_std=0.1)
    gen = torch.Generator(device="cpu").manual_seed(7)
    dST = torch.randn(x["S0"].shape, generator=gen).cuda()
    dRT = torch.randn(x["R0"].shape, generator=gen).cuda()
    _condition(x, clip, dtype)
    d = _gpu(x, clip, dST, dRT)
    ref = _ref(x, clip, dST, dRT)
    for name in GRADS:
        assert_close(d[name], ref[name], dtype, name)


def test_bwd_zero_upstream_state_grads_and_no_init_state():
    x = make_inputs(1, 100, 2, 128, dtype="bf16", nonzero_state=False, with_grad_out=True,
                    device="cuda")
    _condition(x, 1.0, "bf16")
    d = _gpu(x, 1.0)
    ref = _ref(x, 1.0)
    for name in GRADS:
        assert_close(d[name], ref[name], "bf16", name)


@pytest.mark.parametrize("dtype", ["bf16", "f32"])
@pytest.mark.parametrize("D", [64, 128])
def test_bwd_query_scale(dtype, D):
    """The query scale (e.g. 1/sqrt(d_k)): dq is w.r.t. the unscaled query."""
    scale = D ** -0.5
    x = make_inputs(2, 130, 2, D, dtype=dtype, nonzero_state=True, with_grad_out=True,
                    device="cuda", state_std=0.1)
    gen = torch.Generator(device="cpu").manual_seed(11)
    dST = torch.randn(x["S0"].shape, generator=gen).cuda()
    dRT = torch.randn(x["R0"].shape, generator=gen).cuda()
    _condition(x, 1.0, dtype)
    d = _gpu(x, 1.0, dST, dRT, scale=scale)
    ref = _ref(x, 1.0, dST, dRT, scale=scale)
    for name in GRADS:
        assert_close(d[name], ref[name], dtype, name)


@pytest.mark.parametrize("clip", [0.3, float("inf")])
def test_bwd_clip_values(clip):
    x = make_inputs(1, 130, 2, 128, dtype="bf16", nonzero_state=True, with_grad_out=True,
                    device="cuda", state_std=0.1)
    _condition(x, clip, "bf16")
    d = _gpu(x, clip)
    ref = _ref(x, clip)
    for name in GRADS:
        assert_close(d[name], ref[name], "bf16", name)


def test_bwd_reuses_forward_chunk_states():
    """Passing the forward's chunk-start states gives the same gradients as
    letting the backward recompute them."""
    x = make_inputs(2, 192, 2, 128, dtype="bf16", nonzero_state=True, with_grad_out=True,
                    device="cuda", state_std=0.1)
    o, ST, RT, Sc, Rc = rdn.rdn_fwd(*(x[n] for n in NAMES), clip=1.0, S0=x["S0"], R0=x["R0"],
                                    return_chunk_states=True)
    d1 = _gpu(x, 1.0, S_chunks=Sc, R_chunks=Rc)
    d2 = _gpu(x, 1.0)
    # the per-chunk accumulators sum d_v slices with fp32 atomics, so two runs
    # may differ by fp32 rounding, i.e. by one bf16 ulp after the final store
    for name in GRADS:
        torch.testing.assert_close(d1[name].float(), d2[name].float(), atol=1e-5, rtol=8e-3)


@pytest.mark.parametrize("dtype,D", [("bf16", 128), ("bf16", 64), ("f32", 128)])
def test_bwd_reuses_forward_records(dtype, D):
    """Passing the forward's workspace (its per-chunk matrices) with its chunk
    states gives the same gradients as recomputing them, and matches the
    oracle."""
    x = make_inputs(2, 150, 2, D, dtype=dtype, nonzero_state=True, with_grad_out=True,
                    device="cuda", state_std=0.1)
    _condition(x, 1.0, dtype)
    nb = rdn.workspace_bytes("rdn_fwd", 2, 150, 2, D,
                             torch.bfloat16 if dtype == "bf16" else torch.float32)
    wsf = torch.empty(nb, dtype=torch.uint8, device="cuda")
    o, ST, RT, Sc, Rc = rdn.rdn_fwd(*(x[n] for n in NAMES), clip=1.0, S0=x["S0"], R0=x["R0"],
                                    return_chunk_states=True, workspace=wsf)
    d1 = _gpu(x, 1.0, S_chunks=Sc, R_chunks=Rc, fwd_workspace=wsf)
    d2 = _gpu(x, 1.0, S_chunks=Sc, R_chunks=Rc)
    ref = _ref(x, 1.0)
    for name in GRADS:
        torch.testing.assert_close(d1[name].float(), d2[name].float(), atol=1e-5, rtol=8e-3)
        assert_close(d1[name], ref[name], dtype, name)


@pytest.mark.parametrize("variant", ["rdn", "rla"])
@pytest.mark.parametrize("dtype,D,T", [("bf16", 128, 150), ("bf16", 128, 1), ("bf16", 64, 150),
                                       ("f32", 128, 150)])
def test_bwd_uses_forward_saved_intermediates(variant, dtype, D, T):
    """A forward run with save_for_bwd keeps E, E2 and the clip mask; the
    backward that reads them matches the one that recomputes them, and the
    oracle."""
    ov = oracle.RDN if variant == "rdn" else oracle.RLA
    x = make_inputs(2, T, 2, D, dtype=dtype, nonzero_state=True, with_grad_out=True,
                    device="cuda", state_std=0.1)
    _condition(x, 1.0, dtype, variant=ov)
    tdt = torch.bfloat16 if dtype == "bf16" else torch.float32
    wsf = torch.empty(rdn.workspace_bytes(f"{variant}_fwd", 2, T, 2, D, tdt, save_for_bwd=True),
                      dtype=torch.uint8, device="cuda")
    fwd = rdn.rdn_fwd if variant == "rdn" else rdn.rla_fwd
    o, ST, RT, Sc, Rc = fwd(*(x[n] for n in NAMES), clip=1.0, S0=x["S0"], R0=x["R0"],
                            return_chunk_states=True, workspace=wsf, save_for_bwd=True)
    d1 = _gpu(x, 1.0, S_chunks=Sc, R_chunks=Rc, fwd_workspace=wsf, fwd_saved=True,
              variant=variant)
    d2 = _gpu(x, 1.0, S_chunks=Sc, R_chunks=Rc, variant=variant)
    ref = _ref(x, 1.0, variant=ov)
    for name in GRADS:
        torch.testing.assert_close(d1[name].float(), d2[name].float(), atol=1e-5, rtol=8e-3)
        assert_close(d1[name], ref[name], dtype, name)


def test_dalpha_from_dg():
    """dL/dalpha = dg / alpha (the library returns the log-decay gradient)."""
    x = make_inputs(1, 70, 1, 64, dtype="f32", nonzero_state=True, with_grad_out=True,
                    device="cuda", state_std=0.1)
    _condition(x, 1.0, "f32")
    d = _gpu(x, 1.0)
    ref = _ref(x, 1.0)
    alpha = np.exp(as64(x["g"]))
    np.testing.assert_allclose(as64(d["dg"]) / alpha, ref["dg"] / alpha, atol=2e-4, rtol=1e-4)


# ------------------------------------------------------------------ rla_bwd
@pytest.mark.parametrize("dtype", ["bf16", "f32"])
@pytest.mark.parametrize("D", [64, 128])
@pytest.mark.parametrize("T", [1, 64, 65, 200])
def test_rla_bwd_small(dtype, D, T):
    """rla_bwd against the oracle's RLA back-propagation through time (nonzero
    states, upstream state gradients, several chunks and a ragged tail)."""
    clip = 1.0
    x = make_inputs(2, T, 2, D, dtype=dtype, nonzero_state=True, with_grad_out=True,
                    device="cuda", state_std=0.1)
    gen = torch.Generator(device="cpu").manual_seed(17)
    dST = torch.randn(x["S0"].shape, generator=gen).cuda()
    dRT = torch.randn(x["R0"].shape, generator=gen).cuda()
    _condition(x, clip, dtype, variant=oracle.RLA)
    d = _gpu(x, clip, dST, dRT, variant="rla")
    ref = _ref(x, clip, dST, dRT, variant=oracle.RLA)
    for name in GRADS:
        assert_close(d[name], ref[name], dtype, name)


@pytest.mark.parametrize("clip", [0.3, float("inf")])
def test_rla_bwd_clip_and_scale(clip):
    scale = 128 ** -0.5
    x = make_inputs(1, 130, 2, 128, dtype="bf16", nonzero_state=True, with_grad_out=True,
                    device="cuda", state_std=0.1)
    _condition(x, clip, "bf16", variant=oracle.RLA)
    d = _gpu(x, clip, variant="rla", scale=scale)
    ref = _ref(x, clip, variant=oracle.RLA, scale=scale)
    for name in GRADS:
        assert_close(d[name], ref[name], "bf16", name)


@pytest.mark.parametrize("dtype,D", [("bf16", 128), ("f32", 64)])
def test_rla_bwd_reuses_forward(dtype, D):
    """rla_bwd reading rla_fwd's chunk-start states and records gives the
    recomputing backward's gradients, and the oracle's."""
    x = make_inputs(2, 150, 2, D, dtype=dtype, nonzero_state=True, with_grad_out=True,
                    device="cuda", state_std=0.1)
    _condition(x, 1.0, dtype, variant=oracle.RLA)
    nb = rdn.workspace_bytes("rla_fwd", 2, 150, 2, D,
                             dtype=torch.bfloat16 if dtype == "bf16" else torch.float32)
    ws = torch.empty(nb, dtype=torch.uint8, device="cuda")
    _, _, _, Sc, Rc = rdn.rla_fwd(*(x[n] for n in NAMES), clip=1.0, S0=x["S0"], R0=x["R0"],
                                  return_chunk_states=True, workspace=ws)
    d1 = _gpu(x, 1.0, variant="rla", S_chunks=Sc, R_chunks=Rc, fwd_workspace=ws)
    d2 = _gpu(x, 1.0, variant="rla")
    ref = _ref(x, 1.0, variant=oracle.RLA)
    for name in GRADS:
        torch.testing.assert_close(d1[name].float(), d2[name].float(), atol=1e-5, rtol=8e-3)
        assert_close(d1[name], ref[name], dtype, name)


# ------------------------------------------------------------- tied gates
@pytest.mark.parametrize("variant,dtype,D", [("rdn", "bf16", 128), ("rdn", "f32", 64),
                                             ("rla", "bf16", 128)])
def test_tied_gates(variant, dtype, D):
    """RDN_FLAG_TIED_GAMMA: the forward with gamma omitted equals the oracle at
    gamma = beta, and the backward returns the shared gate's gradient in dbeta
    (dgamma not requested: the library keeps the gamma part in its workspace)."""
    ov = oracle.RDN if variant == "rdn" else oracle.RLA
    x = make_inputs(2, 130, 2, D, dtype=dtype, nonzero_state=True, with_grad_out=True,
                    device="cuda", state_std=0.1)
    x["gamma"] = x["beta"]
    _condition(x, 1.0, dtype, variant=ov)
    fwd = rdn.rdn_fwd if variant == "rdn" else rdn.rla_fwd
    o, ST, RT = fwd(*(x[n] for n in NAMES[:5]), None, clip=1.0, S0=x["S0"], R0=x["R0"],
                    tied_gamma=True)
    ref_o, ref_ST, _ = oracle.fwd(ov, *(as64(x[n]) for n in NAMES), 1.0, as64(x["S0"]),
                                  as64(x["R0"]))
    assert_close(o, ref_o, dtype, "o")
    assert_close(ST, ref_ST, dtype, "ST")
    B, T, H = x["g"].shape
    out = dict(dq=torch.empty_like(x["q"]), dk=torch.empty_like(x["k"]), dv=torch.empty_like(x["v"]),
               dg=torch.empty(B, T, H, device="cuda"), dbeta=torch.empty(B, T, H, device="cuda"),
               dS0=torch.empty_like(x["S0"]), dR0=torch.empty_like(x["R0"]))
    bwd = rdn.rdn_bwd if variant == "rdn" else rdn.rla_bwd
    d = bwd(*(x[n] for n in NAMES[:5]), None, x["dO"], clip=1.0, S0=x["S0"], R0=x["R0"],
            out=out, tied_gamma=True)
    torch.cuda.synchronize()
    ref = _ref(x, 1.0, variant=ov)
    assert_close(d["dbeta"], ref["dbeta"] + ref["dgamma"], dtype, "dbeta (tied)")
    for name in ("dq", "dk", "dv", "dg", "dS0", "dR0"):
        assert_close(d[name], ref[name], dtype, name)


@pytest.mark.parametrize("variant", ["rdn", "rla"])
@pytest.mark.parametrize("T", [1, 65, 200])
def test_bwd_f32_out(variant, T):
    """RDN_FLAG_F32_OUT in the backward: dq, dk, dv in fp32 are the values the
    bf16 results round, and they meet the plain 2e-2 RMS bound."""
    ov = oracle.RDN if variant == "rdn" else oracle.RLA
    x = make_inputs(2, T, 2, 128, dtype="bf16", nonzero_state=True, with_grad_out=True,
                    device="cuda", state_std=0.1)
    _condition(x, 1.0, "bf16", variant=ov)
    d = _gpu(x, 1.0, variant=variant)
    d32 = _gpu(x, 1.0, variant=variant, f32_out=True)
    ref = _ref(x, 1.0, variant=ov)
    for name in GRADS:
        if name in ("dq", "dk", "dv"):
            assert d32[name].dtype == torch.float32
            assert torch.equal(d32[name].to(torch.bfloat16), d[name]), name
            assert_close(d32[name], ref[name], "bf16", f"{name} (fp32 out)")
        else:
            assert torch.equal(d32[name], d[name]), name


@pytest.mark.parametrize("variant", ["rdn", "rla"])
@pytest.mark.parametrize("saved", [False, True])
def test_bounded_wait_gives_up_cleanly_bwd(variant, saved, monkeypatch):
    """A device wait of the backward that runs out: with
    RDN_FAULT_INJECT=device_wait_bwd the backward chain skips its first MMA
    completion signal, every thread's bounded wait on it gives up (~5 ms), and
    the CTA records RDN_ERR_TIMEOUT, waits for its MMAs and copies still in
    flight, frees its TMEM and returns (bwd_post then runs on what it has).
    The context stays usable: the next backward matches the oracle and leaves
    the status word at 0."""
    x = make_inputs(2, 200, 2, 128, dtype="bf16", nonzero_state=True, with_grad_out=True,
                    device="cuda", state_std=0.1)
    ov = oracle.RDN if variant == "rdn" else oracle.RLA
    _condition(x, 1.0, "bf16", variant=ov)
    kw = {}
    if saved:  # the forward's chunk states, records and saved intermediates
        wsf = torch.empty(rdn.workspace_bytes(f"{variant}_fwd", 2, 200, 2, 128, save_for_bwd=True),
                          dtype=torch.uint8, device="cuda")
        fwd = rdn.rdn_fwd if variant == "rdn" else rdn.rla_fwd
        _, _, _, Sc, Rc = fwd(*(x[n] for n in NAMES), clip=1.0, S0=x["S0"], R0=x["R0"],
                              return_chunk_states=True, workspace=wsf, save_for_bwd=True)
        kw = dict(S_chunks=Sc, R_chunks=Rc, fwd_workspace=wsf, fwd_saved=True)
    rdn.device_status()  # whatever an earlier test left
    monkeypatch.setenv("RDN_FAULT_INJECT", "device_wait_bwd")
    _gpu(x, 1.0, variant=variant, **kw)
    assert rdn.device_status() == 4  # RDN_ERR_TIMEOUT
    monkeypatch.delenv("RDN_FAULT_INJECT")
    d = _gpu(x, 1.0, variant=variant, **kw)
    assert rdn.device_status() == 0
    ref = _ref(x, 1.0, variant=ov)
    for name in GRADS:
        assert_close(d[name], ref[name], "bf16", name)
