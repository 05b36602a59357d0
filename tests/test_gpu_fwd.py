"""Parity of rla_fwd / rdn_fwd with the fp64 oracle, through the C ABI.

Small cases are compared element by element in full; the full-size
workloads, every head, are in tests/test_gpu_full_size.py."""
import numpy as np
import pytest
import torch

import oracle
import paper_2509_25223_gb300 as rdn
from rdn_synthetic import WORKLOADS, make_inputs, make_workload_inputs
from tests.parity_util import as64, assert_close, err_stats

pytestmark = pytest.mark.gpu

NAMES = ("q", "k", "v", "g", "beta", "gamma")


def _gpu(variant, x, clip=1.0, **kw):
    fn = rdn.rdn_fwd if variant == "rdn" else rdn.rla_fwd
    out = fn(*(x[n] for n in NAMES), clip=clip, S0=x["S0"], R0=x["R0"], **kw)
    torch.cuda.synchronize()
    return out


def _ref(variant, x, clip=1.0, heads=None, scale=1.0):
    """Oracle on all heads, or on the listed (b, h) pairs (returns stacked)."""
    v = oracle.RDN if variant == "rdn" else oracle.RLA
    if heads is None:
        return oracle.fwd(v, *(as64(x[n]) for n in NAMES), clip, as64(x["S0"]), as64(x["R0"]),
                          scale=scale)
    outs = []
    for b, h in heads:
        sl = {n: as64(x[n][b:b + 1, :, h:h + 1]) for n in NAMES}
        S0 = None if x["S0"] is None else as64(x["S0"][b:b + 1, h:h + 1])
        R0 = None if x["R0"] is None else as64(x["R0"][b:b + 1, h:h + 1])
        outs.append(oracle.fwd(v, *(sl[n] for n in NAMES), clip, S0, R0))
    return outs


def test_rla_fwd_f32_workload():
    """RLA, B=1 H=2 T=256 D=64, fp32, zero states, clip 1: every element."""
    w = WORKLOADS["rla_fwd_f32_B1H2T256D64"]
    x = make_workload_inputs(w, device="cuda")
    o, ST, RT = _gpu("rla", x)
    oref, Sref, Rref = _ref("rla", x)
    assert_close(o, oref, "f32", "o")
    assert_close(ST, Sref, "f32", "ST")
    assert_close(RT, Rref, "f32", "RT")


@pytest.mark.parametrize("variant", ["rdn", "rla"])
@pytest.mark.parametrize("dtype", ["bf16", "f32"])
@pytest.mark.parametrize("D", [64, 128])
@pytest.mark.parametrize("T", [1, 2, 3, 7, 8, 63, 64, 65, 200])
def test_fwd_small(variant, dtype, D, T):
    """Several chunks plus a ragged tail, nonzero initial states."""
    x = make_inputs(2, T, 3, D, dtype=dtype, nonzero_state=True, device="cuda", state_std=0.1)
    o, ST, RT = _gpu(variant, x)
    oref, Sref, Rref = _ref(variant, x)
    assert_close(o, oref, dtype, "o")
    assert_close(ST, Sref, dtype, "ST")
    assert_close(RT, Rref, dtype, "RT")


@pytest.mark.parametrize("variant", ["rdn", "rla"])
@pytest.mark.parametrize("dtype", ["bf16", "f32"])
@pytest.mark.parametrize("D", [64, 128])
def test_fwd_query_scale(variant, dtype, D):
    """The query scale (e.g. 1/sqrt(d_k)) enters every read-out."""
    scale = D ** -0.5
    x = make_inputs(2, 130, 2, D, dtype=dtype, nonzero_state=True, device="cuda", state_std=0.1)
    o, ST, RT = _gpu(variant, x, scale=scale)
    oref, Sref, Rref = _ref(variant, x, scale=scale)
    assert_close(o, oref, dtype, "o")
    assert_close(ST, Sref, dtype, "ST")
    assert_close(RT, Rref, dtype, "RT")


@pytest.mark.parametrize("clip", [0.0, 0.25, float("inf")])
def test_rdn_fwd_clip_values(clip):
    x = make_inputs(1, 130, 2, 128, dtype="bf16", nonzero_state=True, device="cuda", state_std=0.1)
    o, ST, RT = _gpu("rdn", x, clip=clip)
    oref, Sref, Rref = _ref("rdn", x, clip=clip)
    assert_close(o, oref, "bf16", "o")
    assert_close(RT, Rref, "bf16", "RT")


def test_fwd_T0_returns_initial_state():
    x = make_inputs(2, 0, 2, 64, dtype="bf16", nonzero_state=True, device="cuda")
    o, ST, RT = _gpu("rdn", x)
    assert o.numel() == 0
    assert torch.equal(ST, x["S0"]) and torch.equal(RT, x["R0"])


def test_chunk_states_and_continuation():
    """S_chunks[c] is the state after 64c tokens, and fwd(T1) -> fwd(T2, S0,
    R0) equals fwd(T1 + T2) (the states are the layer's resume point)."""
    x = make_inputs(1, 192, 2, 128, dtype="bf16", nonzero_state=True, device="cuda", state_std=0.1)
    o, ST, RT, Sc, Rc = _gpu("rdn", x, return_chunk_states=True)
    head = {n: (t[:, :128].contiguous() if t is not None and t.dim() >= 3 and t.shape[1] == 192 else t)
            for n, t in x.items()}
    tail = {n: (t[:, 128:].contiguous() if t is not None and t.dim() >= 3 and t.shape[1] == 192 else t)
            for n, t in x.items()}
    o1, S1, R1 = _gpu("rdn", head)
    torch.testing.assert_close(Sc[:, :, 2], S1, atol=1e-5, rtol=1e-5)
    torch.testing.assert_close(Rc[:, :, 2], R1, atol=1e-5, rtol=1e-5)
    torch.testing.assert_close(Sc[:, :, 0], x["S0"])
    tail["S0"], tail["R0"] = S1, R1
    o2, S2, R2 = _gpu("rdn", tail)
    torch.testing.assert_close(torch.cat([o1, o2], 1).float(), o.float(), atol=2e-2, rtol=0)
    torch.testing.assert_close(S2, ST, atol=1e-4, rtol=1e-4)


def test_device_status_clear_after_normal_calls():
    """No bounded wait gives up on a normal forward and backward: the device
    status word reads 0 (and reading clears it)."""
    x = make_inputs(2, 200, 2, 128, dtype="bf16", nonzero_state=True, with_grad_out=True,
                    device="cuda", state_std=0.1)
    rdn.device_status()  # whatever an earlier test left
    for variant in ("rdn", "rla"):
        fwd = rdn.rdn_fwd if variant == "rdn" else rdn.rla_fwd
        bwd = rdn.rdn_bwd if variant == "rdn" else rdn.rla_bwd
        fwd(*(x[n] for n in NAMES), clip=1.0, S0=x["S0"], R0=x["R0"])
        bwd(*(x[n] for n in NAMES), x["dO"], clip=1.0, S0=x["S0"], R0=x["R0"])
        assert rdn.device_status() == 0, variant


@pytest.mark.parametrize("variant", ["rdn", "rla"])
@pytest.mark.parametrize("T", [1, 65, 200])
def test_fwd_f32_out(variant, T):
    """RDN_FLAG_F32_OUT: o in fp32 is the value the bf16 result rounds, and it
    meets the plain 2e-2 RMS bound (no store rounding)."""
    x = make_inputs(2, T, 3, 128, dtype="bf16", nonzero_state=True, device="cuda", state_std=0.1)
    o, ST, RT = _gpu(variant, x)
    o32, ST2, RT2 = _gpu(variant, x, f32_out=True)
    assert o32.dtype == torch.float32 and torch.equal(o32.to(torch.bfloat16), o)
    assert torch.equal(ST, ST2) and torch.equal(RT, RT2)
    oref, _, _ = _ref(variant, x)
    assert_close(o32, oref, "bf16", "o (fp32 out)")


@pytest.mark.parametrize("variant", ["rdn", "rla"])
def test_bounded_wait_gives_up_cleanly(variant, monkeypatch):
    """A device wait that runs out: with RDN_FAULT_INJECT=device_wait the
    tensor-core scan skips its first MMA completion signal, so every thread's
    bounded wait on it gives up (after ~5 ms instead of ~1 s).  The kernel
    records RDN_ERR_TIMEOUT in the status word, drains what it has in flight,
    frees its TMEM and returns; the context stays usable: the next calls,
    forward and backward, match the oracle and leave the word at 0."""
    x = make_inputs(2, 200, 2, 128, dtype="bf16", nonzero_state=True, device="cuda",
                    state_std=0.1)
    rdn.device_status()  # whatever an earlier test left
    monkeypatch.setenv("RDN_FAULT_INJECT", "device_wait")
    _gpu(variant, x)
    assert rdn.device_status() == 4  # RDN_ERR_TIMEOUT
    monkeypatch.delenv("RDN_FAULT_INJECT")
    o, ST, RT = _gpu(variant, x)
    assert rdn.device_status() == 0
    oref, Sref, Rref = _ref(variant, x)
    assert_close(o, oref, "bf16", "o")
    assert_close(ST, Sref, "bf16", "ST")
    assert_close(RT, Rref, "bf16", "RT")
