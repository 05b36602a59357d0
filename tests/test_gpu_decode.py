"""Parity of rdn_decode_step (single-token step, states in place) with the
oracle, through the C ABI."""
import numpy as np
import pytest
import torch

import oracle
import paper_2509_25223_gb300 as rdn
from rdn_synthetic import make_decode_inputs, make_inputs
from tests.parity_util import as64, assert_close

pytestmark = pytest.mark.gpu


def _step(x, t, variant, clip=1.0, dtype="bf16"):
    S = x["S"].clone()
    R = x["R"].clone()
    o = rdn.rdn_decode_step(x["q"][t], x["k"][t], x["v"][t], x["g"][t], x["beta"][t],
                            x["gamma"][t], S, R, clip=clip, variant=variant)
    torch.cuda.synchronize()
    ref = oracle.decode_step(oracle.RDN if variant == "rdn" else oracle.RLA,
                             as64(x["q"][t]), as64(x["k"][t]), as64(x["v"][t]), as64(x["g"][t]),
                             as64(x["beta"][t]), as64(x["gamma"][t]), clip, as64(x["S"]),
                             as64(x["R"]))
    return (o, S, R), ref


@pytest.mark.parametrize("variant", ["rdn", "rla"])
@pytest.mark.parametrize("D", [64, 128])
@pytest.mark.parametrize("dtype", ["bf16", "f32"])
def test_decode_small(variant, D, dtype):
    x = make_decode_inputs(5, 3, D, steps=1, device="cuda", state_std=0.3, dtype=dtype)
    (o, S, R), (oref, Sref, Rref) = _step(x, 0, variant)
    tol = "f32" if dtype == "f32" else "bf16"
    assert_close(o, oref, tol, "o")
    assert_close(S, Sref, "f32", "S")  # states are fp32 and updated in fp32
    assert_close(R, Rref, "f32", "R")


def test_decode_full_size_one_step():
    """The bench's workload: N=256, H=16, D=128, fp32 states in place."""
    x = make_decode_inputs(256, 16, 128, steps=1, device="cuda")
    (o, S, R), (oref, Sref, Rref) = _step(x, 0, "rdn")
    assert_close(o, oref, "bf16", "o")
    assert_close(S, Sref, "f32", "S")
    assert_close(R, Rref, "f32", "R")


def test_decode_chain_equals_forward():
    """T successive decode steps reproduce the sequence forward of the oracle."""
    B, T, H, D = 3, 20, 2, 128
    x = make_inputs(B, T, H, D, dtype="bf16", nonzero_state=True, device="cuda", state_std=0.1)
    S, R = x["S0"].clone(), x["R0"].clone()
    outs = []
    for t in range(T):
        outs.append(rdn.rdn_decode_step(x["q"][:, t].contiguous(), x["k"][:, t].contiguous(),
                                        x["v"][:, t].contiguous(), x["g"][:, t].contiguous(),
                                        x["beta"][:, t].contiguous(), x["gamma"][:, t].contiguous(),
                                        S, R))
    torch.cuda.synchronize()
    o = torch.stack(outs, 1)
    oref, Sref, Rref = oracle.rdn_fwd(*(as64(x[n]) for n in ("q", "k", "v", "g", "beta", "gamma")),
                                      1.0, as64(x["S0"]), as64(x["R0"]))
    assert_close(o, oref, "bf16", "o")
    assert_close(S, Sref, "f32", "S")
    assert_close(R, Rref, "f32", "R")


def test_decode_no_clip_and_zero_clip():
    x = make_decode_inputs(4, 2, 128, steps=1, device="cuda", state_std=0.5)
    for clip in (float("inf"), 0.0):
        (o, S, R), (oref, Sref, Rref) = _step(x, 0, "rdn", clip=clip)
        assert_close(o, oref, "bf16", f"o clip={clip}")
        assert_close(R, Rref, "f32", f"R clip={clip}")


@pytest.mark.parametrize("variant", ["rdn", "rla"])
@pytest.mark.parametrize("flags", [rdn.DECAYED_RESIDUAL, rdn.PLAIN_COMBINE, rdn.TANH_RESIDUAL,
                                   rdn.STATELESS_AUX,
                                   rdn.DECAYED_RESIDUAL | rdn.TANH_RESIDUAL | rdn.PLAIN_COMBINE])
@pytest.mark.parametrize("tied", [False, True])
def test_decode_variants(variant, flags, tied):
    """The variant flags and tied gates in the decode step equal one token of
    the oracle's forward with the same variant bits (S0, R0 = the states)."""
    x = make_decode_inputs(5, 3, 128, steps=1, device="cuda", state_std=0.3)
    mods = {rdn.DECAYED_RESIDUAL: oracle.DECAYED, rdn.PLAIN_COMBINE: oracle.PLAIN,
            rdn.TANH_RESIDUAL: oracle.TANH, rdn.STATELESS_AUX: oracle.STATELESS}
    m = sum(o for f, o in mods.items() if flags & f)
    gam = x["beta"][0] if tied else x["gamma"][0]
    S, R = x["S"].clone(), x["R"].clone()
    o = rdn.rdn_decode_step(x["q"][0], x["k"][0], x["v"][0], x["g"][0], x["beta"][0],
                            None if tied else gam, S, R, clip=0.7, variant=variant,
                            tied_gamma=tied, variant_flags=flags)
    torch.cuda.synchronize()
    tok = lambda t: as64(t)[:, None]  # [N,H,...] -> [N,1,H,...]: one token of the forward
    oref, Sref, Rref = oracle.fwd(oracle.RDN if variant == "rdn" else oracle.RLA,
                                  tok(x["q"][0]), tok(x["k"][0]), tok(x["v"][0]), tok(x["g"][0]),
                                  tok(x["beta"][0]), tok(gam), 0.7, as64(x["S"]), as64(x["R"]),
                                  mods=m)
    assert_close(o, oref[:, 0], "bf16", "o")
    assert_close(S, Sref, "f32", "S")
    assert_close(R, Rref, "f32", "R")

