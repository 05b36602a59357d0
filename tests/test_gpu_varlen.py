"""Packed variable-length sequences (rdn_fwd_args.cu_seqlens) through the C ABI.

Sequences in a packed batch are independent recurrences, each starting from
its own initial state, so the reference for sequence s is the oracle run on
that sequence alone (an empty sequence passes its states through).  Besides
the element-wise parity with the oracle, the packed call must give the same
bits as one unpacked call per sequence: the per-sequence arithmetic does not
depend on where a sequence sits in the batch."""
import numpy as np
import pytest
import torch

import oracle
import paper_2509_25223_gb300 as rdn
from rdn_synthetic import make_inputs
from tests.parity_util import as64, assert_close

pytestmark = pytest.mark.gpu

NAMES = ("q", "k", "v", "g", "beta", "gamma")
GRADS = ("dq", "dk", "dv", "dg", "dbeta", "dgamma")
MARGIN = 1e-2
# empty sequences, single tokens, exact chunk multiples and ragged tails
LENS = [0, 1, 63, 64, 65, 150, 0, 130]


def _packed(lens, H, D, dtype, seed=0):
    T = int(sum(lens))
    x = make_inputs(1, T, H, D, dtype=dtype, with_grad_out=True, device="cuda", seed=seed)
    gen = torch.Generator(device="cpu").manual_seed(seed + 11)
    N = len(lens)
    for n in ("S0", "R0", "dST", "dRT"):
        x[n] = (0.1 * torch.randn(N, H, D, D, generator=gen)).cuda()
    cu = np.concatenate([[0], np.cumsum(lens)]).astype(np.int32)
    x["cu"] = torch.from_numpy(cu).cuda()
    x["cu_host"] = cu
    return x


def _seq(x, s, n):
    """Sequence s of the packed inputs as a B = 1 problem (device tensors)."""
    t0, t1 = int(x["cu_host"][s]), int(x["cu_host"][s + 1])
    return x[n][:, t0:t1].clone()  # (own allocation: the library wants 16-byte alignment)


def _condition(x, clip, dtype, variant):
    """Move v so every fp64 clip decision of every sequence has a margin."""
    H = x["q"].shape[2]
    for s in range(len(x["cu_host"]) - 1):
        t0, t1 = int(x["cu_host"][s]), int(x["cu_host"][s + 1])
        if t1 == t0:
            continue
        for h in range(H):
            sl = {n: as64(x[n][:, t0:t1, h:h + 1]) for n in NAMES}
            v2, _ = oracle.clip_margin_condition(variant, sl["q"], sl["k"], sl["v"], sl["g"],
                                                 sl["beta"], sl["gamma"], clip,
                                                 as64(x["S0"][s:s + 1, h:h + 1]),
                                                 as64(x["R0"][s:s + 1, h:h + 1]),
                                                 margin=MARGIN, quant=dtype)
            x["v"][0, t0:t1, h] = torch.from_numpy(v2[0, :, 0]).to(x["v"].dtype).cuda()


def _fwd(variant, x, clip, **kw):
    fn = rdn.rdn_fwd if variant == "rdn" else rdn.rla_fwd
    return fn(*(x[n] for n in NAMES), clip=clip, S0=x["S0"], R0=x["R0"], cu_seqlens=x["cu"],
              **kw)


@pytest.mark.parametrize("variant", ["rdn", "rla"])
@pytest.mark.parametrize("dtype,D", [("bf16", 128), ("f32", 64), ("bf16", 64)])
def test_packed_fwd_matches_oracle_per_sequence(variant, dtype, D):
    clip = 1.0
    x = _packed(LENS, 2, D, dtype)
    o, ST, RT = _fwd(variant, x, clip)
    torch.cuda.synchronize()
    v = oracle.RDN if variant == "rdn" else oracle.RLA
    for s in range(len(LENS)):
        if LENS[s] == 0:  # no tokens: the final states are the initial ones
            assert torch.equal(ST[s], x["S0"][s]) and torch.equal(RT[s], x["R0"][s])
            continue
        oref, Sref, Rref = oracle.fwd(v, *(as64(_seq(x, s, n)) for n in NAMES), clip,
                                      as64(x["S0"][s:s + 1]), as64(x["R0"][s:s + 1]))
        t0, t1 = int(x["cu_host"][s]), int(x["cu_host"][s + 1])
        assert_close(o[:, t0:t1], oref, dtype, f"o[{s}]")
        assert_close(ST[s:s + 1], Sref, dtype, f"ST[{s}]")
        assert_close(RT[s:s + 1], Rref, dtype, f"RT[{s}]")


@pytest.mark.parametrize("variant", ["rdn", "rla"])
@pytest.mark.parametrize("dtype,D", [("bf16", 128), ("f32", 64)])
def test_packed_fwd_bitwise_equals_separate_calls(variant, dtype, D):
    """o, final states and every sequence's chunk-start states equal those of
    an unpacked call on that sequence alone, bit for bit."""
    x = _packed(LENS, 3, D, dtype, seed=3)
    H = 3
    o, ST, RT, Sc, Rc = _fwd(variant, x, 1.0, return_chunk_states=True)
    fn = rdn.rdn_fwd if variant == "rdn" else rdn.rla_fwd
    cbase = 0
    for s, L in enumerate(LENS):
        nc = (L + 63) // 64
        if L == 0:
            continue
        o1, S1, R1, Sc1, Rc1 = fn(*(_seq(x, s, n) for n in NAMES), clip=1.0,
                                  S0=x["S0"][s:s + 1], R0=x["R0"][s:s + 1],
                                  return_chunk_states=True)
        t0, t1 = int(x["cu_host"][s]), int(x["cu_host"][s + 1])
        assert torch.equal(o[:, t0:t1], o1), s
        assert torch.equal(ST[s:s + 1], S1) and torch.equal(RT[s:s + 1], R1), s
        # records of sequence s: (first chunk) * H + h * nc + c
        blk = Sc[cbase * H:(cbase + nc) * H].view(H, nc, D, D)
        assert torch.equal(blk, Sc1[0]), s
        assert torch.equal(Rc[cbase * H:(cbase + nc) * H].view(H, nc, D, D), Rc1[0]), s
        cbase += nc


@pytest.mark.parametrize("variant", ["rdn", "rla"])
@pytest.mark.parametrize("dtype,D", [("bf16", 128), ("f32", 64)])
@pytest.mark.parametrize("reuse", ["recompute", "chunk_states", "saved"])
def test_packed_bwd_matches_oracle_per_sequence(variant, dtype, D, reuse):
    clip = 1.0
    v = oracle.RDN if variant == "rdn" else oracle.RLA
    x = _packed(LENS, 2, D, dtype, seed=5)
    _condition(x, clip, dtype, v)
    kw = {}
    if reuse != "recompute":
        ws = None
        if reuse == "saved":
            nbytes = rdn.workspace_bytes(f"{variant}_fwd", 1, x["q"].shape[1], 2, D,
                                         torch.bfloat16 if dtype == "bf16" else torch.float32,
                                         save_for_bwd=True, cu_seqlens=x["cu"])
            ws = torch.empty(nbytes, dtype=torch.uint8, device="cuda")
        fkw = dict(return_chunk_states=True, workspace=ws)
        if reuse == "saved":
            fkw["save_for_bwd"] = True
        _, _, _, Sc, Rc = _fwd(variant, x, clip, **fkw)
        kw = dict(S_chunks=Sc, R_chunks=Rc)
        if ws is not None:
            kw.update(fwd_workspace=ws, fwd_saved=True)
    fn = rdn.rdn_bwd if variant == "rdn" else rdn.rla_bwd
    d = fn(*(x[n] for n in NAMES), x["dO"], clip=clip, S0=x["S0"], R0=x["R0"], dST=x["dST"],
           dRT=x["dRT"], cu_seqlens=x["cu"], **kw)
    torch.cuda.synchronize()
    for s, L in enumerate(LENS):
        if L == 0:  # no tokens: the upstream state gradients pass through
            assert torch.equal(d["dS0"][s], x["dST"][s]) and torch.equal(d["dR0"][s], x["dRT"][s])
            continue
        ref = oracle.bwd(v, *(as64(_seq(x, s, n)) for n in NAMES), clip,
                         as64(x["S0"][s:s + 1]), as64(x["R0"][s:s + 1]), as64(_seq(x, s, "dO")),
                         as64(x["dST"][s:s + 1]), as64(x["dRT"][s:s + 1]))
        t0, t1 = int(x["cu_host"][s]), int(x["cu_host"][s + 1])
        for name in GRADS:
            assert_close(d[name][:, t0:t1], ref[name], dtype, f"{name}[{s}]")
        assert_close(d["dS0"][s:s + 1], ref["dS0"], dtype, f"dS0[{s}]")
        assert_close(d["dR0"][s:s + 1], ref["dR0"], dtype, f"dR0[{s}]")


def test_packed_all_empty_and_single_sequence():
    """T = 0 with three empty sequences copies the states; one sequence
    covering all tokens equals the unpacked call bit for bit."""
    x = _packed([0, 0, 0], 2, 128, "bf16")
    o, ST, RT = _fwd("rdn", x, 1.0)
    torch.cuda.synchronize()
    assert o.shape[1] == 0
    assert torch.equal(ST, x["S0"]) and torch.equal(RT, x["R0"])
    x = _packed([200], 2, 128, "bf16", seed=9)
    o, ST, RT = _fwd("rdn", x, 1.0)
    o1, S1, R1 = rdn.rdn_fwd(*(x[n] for n in NAMES), clip=1.0, S0=x["S0"], R0=x["R0"])
    assert torch.equal(o, o1) and torch.equal(ST, S1) and torch.equal(RT, R1)


def test_packed_tied_gates():
    """Tied gates with packed sequences: dbeta is the sum of the untied
    gradients of the two gates."""
    x = _packed([70, 0, 129], 2, 128, "bf16", seed=13)
    x["gamma"] = x["beta"].clone()
    _condition(x, 1.0, "bf16", oracle.RDN)
    args = [x[n] for n in NAMES] + [x["dO"]]
    kw = dict(clip=1.0, S0=x["S0"], R0=x["R0"], dST=x["dST"], dRT=x["dRT"], cu_seqlens=x["cu"])
    du = rdn.rdn_bwd(*args, **kw)
    dt = rdn.rdn_bwd(*args, tied_gamma=True, **kw)
    torch.cuda.synchronize()
    assert_close(dt["dbeta"], as64(du["dbeta"]) + as64(du["dgamma"]), "bf16", "dbeta")
    for name in ("dq", "dk", "dv", "dg", "dS0", "dR0"):
        assert_close(dt[name], du[name], "bf16", name)


def test_packed_table_clamped():
    """A table that breaks the ordering is clamped (no fault): entries past
    T read as T, a decreasing entry as its predecessor."""
    x = _packed([40, 30, 50], 2, 64, "f32", seed=17)
    good = x["cu"].clone()
    bad = torch.tensor([5, 40, 10**6, 120], dtype=torch.int32, device="cuda")
    x["cu"] = bad  # reads as [0, 40, 120, 120]: sequences 40, 80, 0 tokens
    o, ST, RT = _fwd("rdn", x, 1.0)
    torch.cuda.synchronize()
    x["cu"] = torch.tensor([0, 40, 120, 120], dtype=torch.int32, device="cuda")
    o2, ST2, RT2 = _fwd("rdn", x, 1.0)
    assert torch.equal(o, o2) and torch.equal(ST, ST2) and torch.equal(RT, RT2)
    x["cu"] = good


def test_packed_bench_shape_sampled():
    """The bench's packed workload (32,768 tokens x 16 heads, d = 128, 15
    log-uniform lengths), fwd + bwd as the bench runs it (chunk states and
    saved intermediates reused); the shortest, a middle and the longest
    sequence checked against the oracle on one head each."""
    from rdn_synthetic import packed_lengths
    lens = packed_lengths(32768)
    T, H, D = sum(lens), 16, 128
    x = make_inputs(1, T, H, D, dtype="bf16", with_grad_out=True, device="cuda", seed=2)
    cu_h = np.concatenate([[0], np.cumsum(lens)]).astype(np.int32)
    x["cu"], x["cu_host"] = torch.from_numpy(cu_h).cuda(), cu_h
    order = np.argsort(lens)
    picks = [(int(order[0]), 3), (int(order[len(lens) // 2]), 9), (int(order[-1]), 14)]
    for s, h in picks:  # margin on the sampled heads' clip decisions
        t0, t1 = int(cu_h[s]), int(cu_h[s + 1])
        sl = {n: as64(x[n][:, t0:t1, h:h + 1]) for n in NAMES}
        v2, _ = oracle.clip_margin_condition(oracle.RDN, *(sl[n] for n in NAMES), 1.0,
                                             margin=MARGIN, quant="bf16")
        x["v"][0, t0:t1, h] = torch.from_numpy(v2[0, :, 0]).to(x["v"].dtype).cuda()
    ws = torch.empty(rdn.workspace_bytes("rdn_fwd", 1, T, H, D, save_for_bwd=True,
                                         cu_seqlens=x["cu"]), dtype=torch.uint8, device="cuda")
    o, ST, RT, Sc, Rc = rdn.rdn_fwd(*(x[n] for n in NAMES), clip=1.0, cu_seqlens=x["cu"],
                                    return_chunk_states=True, workspace=ws, save_for_bwd=True)
    d = rdn.rdn_bwd(*(x[n] for n in NAMES), x["dO"], clip=1.0, cu_seqlens=x["cu"], S_chunks=Sc,
                    R_chunks=Rc, fwd_workspace=ws, fwd_saved=True)
    torch.cuda.synchronize()
    for s, h in picks:
        t0, t1 = int(cu_h[s]), int(cu_h[s + 1])
        sl = {n: as64(x[n][:, t0:t1, h:h + 1]) for n in NAMES + ("dO",)}
        oref, Sref, Rref = oracle.fwd(oracle.RDN, *(sl[n] for n in NAMES), 1.0)
        assert_close(o[:, t0:t1, h:h + 1], oref, "bf16", f"o[{s},{h}]")
        assert_close(ST[s:s + 1, h:h + 1], Sref, "bf16", f"ST[{s},{h}]")
        assert_close(RT[s:s + 1, h:h + 1], Rref, "bf16", f"RT[{s},{h}]")
        ref = oracle.bwd(oracle.RDN, *(sl[n] for n in NAMES), 1.0, None, None, sl["dO"])
        for name in GRADS:
            assert_close(d[name][:, t0:t1, h:h + 1], ref[name], "bf16", f"{name}[{s},{h}]")
        assert_close(d["dS0"][s:s + 1, h:h + 1], ref["dS0"], "bf16", f"dS0[{s},{h}]")
        assert_close(d["dR0"][s:s + 1, h:h + 1], ref["dR0"], "bf16", f"dR0[{s},{h}]")
