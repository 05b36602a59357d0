"""Seeded synthetic inputs for the RLA / RDN layer workloads.

This module is the one place the CUDA path's tests / bench and the CPU oracle
meet: it draws random inputs and holds none of the method's arithmetic.

The workloads stand in for the paper's language-model layers (Appendix C,
Table 6: hidden 2048, 16 heads, head dimension 128).  The paper's training
data is not used; inputs are drawn as follows, in this fixed order, in fp32 on
a CPU ``torch.Generator`` seeded with ``seed`` (or on the target device when
``device_rng`` is set, for sizes where host generation would be slow):

1. q, k ~ N(0,1), then L2-normalised over the head dimension per (b,t,h)
   (the paper normalises q and k before the recurrence, Section 3.3);
2. v ~ N(0,1);
3. x_a ~ N(0,1) and the log-decay g = log(alpha): logsigmoid(x_a) for the
   RLA workload, -softplus(x_a) for the RDN ones (alpha = exp(-softplus(.)),
   the Mamba-2 style parametrisation of Section 3.4 with a = 1, b = 0);
4. beta = sigmoid(N(0,1));  5. gamma = sigmoid(N(0,1));
6. S0, R0 ~ N(0, 0.02^2) where the workload has nonzero initial states;
7. dO ~ N(0,1) for the backward workload.

q, k, v (and dO) are then cast to the workload dtype; gates and states stay
fp32.
"""
from __future__ import annotations

import dataclasses

import torch
import torch.nn.functional as F


@dataclasses.dataclass(frozen=True)
class Workload:
    name: str
    op: str            # "rla_fwd" | "rdn_fwd" | "rdn_fwd_bwd" | "rdn_decode"
    B: int
    H: int
    T: int
    D: int
    dtype: str         # "f32" | "bf16" (q, k, v, o)
    decay: str         # "logsigmoid" | "neg_softplus"
    clip: float = 1.0
    nonzero_state: bool = False
    chunk: int = 64


WORKLOADS = {
    w.name: w
    for w in [
        Workload("rla_fwd_f32_B1H2T256D64", "rla_fwd", 1, 2, 256, 64, "f32", "logsigmoid"),
        Workload("rdn_fwd_bf16_B8H16T2048D128", "rdn_fwd", 8, 16, 2048, 128, "bf16",
                 "neg_softplus"),
        Workload("rdn_fwd_bf16_B2H16T16384D128_state", "rdn_fwd", 2, 16, 16384, 128, "bf16",
                 "neg_softplus", nonzero_state=True),
        Workload("rdn_fwd_bwd_bf16_B8H16T4096D128", "rdn_fwd_bwd", 8, 16, 4096, 128, "bf16",
                 "neg_softplus"),
        Workload("rdn_decode_N256H16D128", "rdn_decode", 256, 16, 1, 128, "bf16",
                 "neg_softplus", nonzero_state=True),
    ]
}

TORCH_DTYPE = {"f32": torch.float32, "bf16": torch.bfloat16}


def make_inputs(B, T, H, D, dtype="bf16", decay="neg_softplus", nonzero_state=False,
                with_grad_out=False, seed=0, device="cpu", device_rng=False, Dv=None,
                state_std=0.02):
    """Draw one batch of inputs in the recipe's order.

    Returns a dict of tensors on `device`: q, k [B,T,H,D]; v [B,T,H,Dv];
    g, beta, gamma [B,T,H] fp32; S0, R0 [B,H,D,Dv] fp32 or None; dO
    [B,T,H,Dv] when with_grad_out."""
    Dv = D if Dv is None else Dv
    gen_dev = device if device_rng else "cpu"
    gen = torch.Generator(device=gen_dev)
    gen.manual_seed(seed)

    def randn(*shape):
        return torch.randn(*shape, generator=gen, device=gen_dev, dtype=torch.float32)

    q = F.normalize(randn(B, T, H, D), dim=-1)
    k = F.normalize(randn(B, T, H, D), dim=-1)
    v = randn(B, T, H, Dv)
    xa = randn(B, T, H)
    g = F.logsigmoid(xa) if decay == "logsigmoid" else -F.softplus(xa)
    beta = torch.sigmoid(randn(B, T, H))
    gamma = torch.sigmoid(randn(B, T, H))
    S0 = R0 = None
    if nonzero_state:
        S0 = randn(B, H, D, Dv) * state_std
        R0 = randn(B, H, D, Dv) * state_std
    dO = randn(B, T, H, Dv) if with_grad_out else None
    td = TORCH_DTYPE[dtype]
    out = dict(q=q.to(td), k=k.to(td), v=v.to(td), g=g, beta=beta, gamma=gamma,
               S0=S0, R0=R0, dO=None if dO is None else dO.to(td))
    return {n: (None if t is None else t.to(device).contiguous()) for n, t in out.items()}


def make_workload_inputs(w: Workload, seed=0, device="cpu", device_rng=False, **over):
    """Inputs for a named workload; keyword overrides (B, T, ...) shrink it."""
    p = dict(B=w.B, T=w.T, H=w.H, D=w.D, dtype=w.dtype, decay=w.decay,
             nonzero_state=w.nonzero_state, with_grad_out=(w.op == "rdn_fwd_bwd"))
    p.update(over)
    return make_inputs(seed=seed, device=device, device_rng=device_rng, **p)


def make_decode_inputs(N, H, D, steps=1, seed=0, device="cpu", device_rng=False,
                       state_std=0.02, dtype="bf16"):
    """Decode workload: states S, R [N,H,D,D] fp32 ~ N(0, state_std^2) and
    `steps` fresh single-token draws (q, k [steps,N,H,D], v [steps,N,H,D]
    in `dtype`; g, beta, gamma [steps,N,H] fp32), same recipe as above."""
    gen_dev = device if device_rng else "cpu"
    gen = torch.Generator(device=gen_dev)
    gen.manual_seed(seed)

    def randn(*shape):
        return torch.randn(*shape, generator=gen, device=gen_dev, dtype=torch.float32)

    S = randn(N, H, D, D) * state_std
    R = randn(N, H, D, D) * state_std
    q = F.normalize(randn(steps, N, H, D), dim=-1)
    k = F.normalize(randn(steps, N, H, D), dim=-1)
    v = randn(steps, N, H, D)
    g = -F.softplus(randn(steps, N, H))
    beta = torch.sigmoid(randn(steps, N, H))
    gamma = torch.sigmoid(randn(steps, N, H))
    td = TORCH_DTYPE[dtype]
    out = dict(S=S, R=R, q=q.to(td), k=k.to(td), v=v.to(td), g=g, beta=beta, gamma=gamma)
    return {n: t.to(device).contiguous() for n, t in out.items()}


def packed_lengths(total, lo=64, hi=8192, seed=1234):
    """Sequence lengths for a packed batch of `total` tokens: log-uniform in
    [lo, hi] from a seeded numpy generator, the last one cut to fill the row
    (a pretraining-style mix of short and long documents)."""
    import numpy as np
    rng = np.random.default_rng(seed)
    lens, tot = [], 0
    while tot < total:
        L = min(int(np.exp(rng.uniform(np.log(lo), np.log(hi)))), total - tot)
        lens.append(L)
        tot += L
    return lens
