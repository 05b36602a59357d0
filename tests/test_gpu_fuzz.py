"""Seeded random configurations of the whole API against the oracle.

Each case draws: RLA or RDN; fp32 or bf16; d = 64 or 128; a batch of equal
sequences or packed sequences of random lengths (empty ones included); the
clip threshold (0, 0.3, 1, inf); the query scale; tied gates; a random set of
the variant flags; initial states and upstream state gradients present or
not (every third case on the tensor-core path).  The forward and the
backward (with the forward's chunk states reused half of the time) are
compared with the oracle sequence by sequence."""
import numpy as np
import pytest
import torch

import oracle
import paper_2509_25223_gb300 as rdn
from rdn_synthetic import make_inputs
from tests.parity_util import as64, assert_close

pytestmark = pytest.mark.gpu

NAMES = ("q", "k", "v", "g", "beta", "gamma")
TO_ORACLE = {rdn.DECAYED_RESIDUAL: oracle.DECAYED, rdn.PLAIN_COMBINE: oracle.PLAIN,
             rdn.TANH_RESIDUAL: oracle.TANH, rdn.STATELESS_AUX: oracle.STATELESS}


def _case(seed):
    rng = np.random.default_rng(1000 + seed)
    c = dict(variant=str(rng.choice(["rdn", "rla"])), dtype=str(rng.choice(["f32", "bf16"])),
             D=int(rng.choice([64, 128])), H=int(rng.integers(1, 4)),
             clip=float(rng.choice([0.0, 0.3, 1.0, np.inf])),
             scale=float(rng.choice([1.0, 0.5])), tied=bool(rng.random() < 0.3),
             flags=int(sum(f for f in TO_ORACLE if rng.random() < 0.25)),
             states=bool(rng.random() < 0.6), dstates=bool(rng.random() < 0.5),
             reuse=bool(rng.random() < 0.5))
    if seed % 3 == 0:  # every third case on the tensor-core path (RDN, bf16, d = 128)
        c.update(variant="rdn", dtype="bf16", D=128, flags=0)
    if rng.random() < 0.4:  # packed sequences
        n = int(rng.integers(1, 5))
        c["lens"] = [int(x) for x in rng.choice([0, 1, 37, 64, 65, 130, 200], size=n)]
        c["B"], c["T"] = 1, sum(c["lens"])
    else:
        c["lens"] = None
        c["B"], c["T"] = int(rng.integers(1, 3)), int(rng.choice([1, 50, 64, 129, 257]))
    return c


@pytest.mark.parametrize("seed", range(48))
def test_fuzz(seed):
    c = _case(seed)
    variant, dtype, D, H, B, T = c["variant"], c["dtype"], c["D"], c["H"], c["B"], c["T"]
    ov = oracle.RDN if variant == "rdn" else oracle.RLA
    mods = sum(o for f, o in TO_ORACLE.items() if c["flags"] & f)
    x = make_inputs(B, T, H, D, dtype=dtype, with_grad_out=True, device="cuda", seed=seed)
    if c["tied"]:
        x["gamma"] = x["beta"]
    lens = c["lens"] if c["lens"] is not None else [T] * B
    N = len(lens)
    gen = torch.Generator(device="cpu").manual_seed(seed)
    st = lambda: (0.1 * torch.randn(N, H, D, D, generator=gen)).cuda()
    S0, R0 = (st(), st()) if c["states"] else (None, None)
    dST, dRT = (st(), st()) if c["dstates"] else (None, None)
    cu = None
    if c["lens"] is not None:
        cu_h = np.concatenate([[0], np.cumsum(lens)]).astype(np.int32)
        cu = torch.from_numpy(cu_h).cuda()
    spans = []  # (row b, first token, last token, sequence index)
    for s, L in enumerate(lens):
        b, t0 = (0, int(sum(lens[:s]))) if c["lens"] is not None else (s, 0)
        spans.append((b, t0, t0 + L, s))
    # clip decisions away from c, per sequence and head
    for b, t0, t1, s in spans:
        if t1 == t0:
            continue
        for h in range(H):
            sl = {n: as64(x[n][b:b + 1, t0:t1, h:h + 1]) for n in NAMES}
            v2, _ = oracle.clip_margin_condition(
                ov, *(sl[n] for n in NAMES), c["clip"],
                None if S0 is None else as64(S0[s:s + 1, h:h + 1]),
                None if R0 is None else as64(R0[s:s + 1, h:h + 1]), scale=c["scale"],
                margin=1e-2, quant=dtype, mods=mods)
            x["v"][b, t0:t1, h] = torch.from_numpy(v2[0, :, 0]).to(x["v"].dtype).cuda()
    gam = None if c["tied"] else x["gamma"]
    kw = dict(clip=c["clip"], S0=S0, R0=R0, scale=c["scale"], tied_gamma=c["tied"],
              variant_flags=c["flags"], cu_seqlens=cu)
    fwd = rdn.rdn_fwd if variant == "rdn" else rdn.rla_fwd
    o, ST, RT, Sc, Rc = fwd(x["q"], x["k"], x["v"], x["g"], x["beta"], gam,
                            return_chunk_states=True, **kw)
    bwd = rdn.rdn_bwd if variant == "rdn" else rdn.rla_bwd
    out = dict(dq=torch.empty_like(x["q"]), dk=torch.empty_like(x["k"]),
               dv=torch.empty_like(x["v"]), dg=torch.empty_like(x["g"]),
               dbeta=torch.empty_like(x["g"]), dS0=torch.empty(N, H, D, D, device="cuda"),
               dR0=torch.empty(N, H, D, D, device="cuda"))
    if not c["tied"]:
        out["dgamma"] = torch.empty_like(x["g"])
    extra = dict(S_chunks=Sc, R_chunks=Rc) if c["reuse"] else {}
    d = bwd(x["q"], x["k"], x["v"], x["g"], x["beta"], gam, x["dO"], dST=dST, dRT=dRT, out=out,
            **kw, **extra)
    torch.cuda.synchronize()
    for b, t0, t1, s in spans:
        sl = {n: as64(x[n][b:b + 1, t0:t1]) for n in NAMES + ("dO",)}
        s0 = None if S0 is None else as64(S0[s:s + 1])
        r0 = None if R0 is None else as64(R0[s:s + 1])
        tag = f"{c} seq {s}"
        if t1 == t0:
            z = torch.zeros(H, D, D, device="cuda")
            assert torch.equal(ST[s], z if S0 is None else S0[s]), tag
            assert torch.equal(d["dS0"][s], z if dST is None else dST[s]), tag
            continue
        oref, Sref, Rref = oracle.fwd(ov, *(sl[n] for n in NAMES), c["clip"], s0, r0,
                                      scale=c["scale"], mods=mods)
        assert_close(o[b:b + 1, t0:t1], oref, dtype, "o " + tag)
        assert_close(ST[s:s + 1], Sref, dtype, "ST " + tag)
        assert_close(RT[s:s + 1], Rref, dtype, "RT " + tag)
        ref = oracle.bwd(ov, *(sl[n] for n in NAMES), c["clip"], s0, r0, sl["dO"],
                         None if dST is None else as64(dST[s:s + 1]),
                         None if dRT is None else as64(dRT[s:s + 1]), scale=c["scale"], mods=mods)
        if c["tied"]:
            ref["dbeta"] = ref["dbeta"] + ref["dgamma"]
        for name in ("dq", "dk", "dv", "dg", "dbeta") + (() if c["tied"] else ("dgamma",)):
            assert_close(d[name][b:b + 1, t0:t1], ref[name], dtype, f"{name} {tag}")
        assert_close(d["dS0"][s:s + 1], ref["dS0"], dtype, "dS0 " + tag)
        assert_close(d["dR0"][s:s + 1], ref["dR0"], dtype, "dR0 " + tag)
