"""Pins for the fp64 oracle: checks against what the paper and mathematics fix,
not against the oracle itself (CPU only).

Each test names the passage it follows.  Together they are chosen so that a
dropped term, a wrong sign, a wrong time index (S_{t-1} vs S_t, R_{t-1} vs
R_t) or a transposed state in the oracle fails at least one of them.
"""
import os

import numpy as np
import pytest
import torch

import oracle
from oracle import RDN, RLA
from tests.chunk_algebra import chunk_fwd
from rdn_synthetic import make_inputs

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _inputs(B=2, T=19, H=2, D=8, Dv=None, nonzero=True, seed=0, decay="neg_softplus"):
    x = make_inputs(B, T, H, D, dtype="f32", decay=decay, nonzero_state=nonzero,
                    with_grad_out=True, seed=seed, Dv=Dv, state_std=0.3)
    return {n: (None if t is None else t.double().numpy()) for n, t in x.items()}


def _fwd(variant, x, c=1.0, **kw):
    return oracle.fwd(variant, x["q"], x["k"], x["v"], x["g"], x["beta"], x["gamma"], c,
                      x["S0"], x["R0"], **kw)


# ---------------------------------------------------------------- P1: T = 1
@pytest.mark.parametrize("variant", [RLA, RDN])
def test_T1_closed_form(variant):
    """Section 3.4 at t = 1: r = clip(v - S0^T k); o = a S0^T q + gam R_1^T q with
    R_1 = a R0 (- a gam k (R0^T k)^T for RDN) + gam k r^T."""
    x = _inputs(B=1, T=1, H=1, D=6, Dv=5)
    q, k, v = x["q"][0, 0, 0], x["k"][0, 0, 0], x["v"][0, 0, 0] * 3.0
    a = np.exp(x["g"][0, 0, 0])
    b, gm = x["beta"][0, 0, 0], x["gamma"][0, 0, 0]
    S0, R0 = x["S0"][0, 0], x["R0"][0, 0]
    c = 0.7
    r = np.clip(v - S0.T @ k, -c, c)
    if variant == RDN:
        R1 = a * R0 - a * gm * np.outer(k, R0.T @ k) + gm * np.outer(k, r)
        S1 = a * S0 - a * b * np.outer(k, S0.T @ k) + b * np.outer(k, v)
    else:
        R1 = a * R0 + gm * np.outer(k, r)
        S1 = a * S0 + b * np.outer(k, v)
    o_exp = a * S0.T @ q + gm * R1.T @ q
    xx = dict(x)
    xx["v"] = (v * 1.0)[None, None, None]
    o, ST, RT = _fwd(variant, xx, c=c)
    np.testing.assert_allclose(o[0, 0, 0], o_exp, rtol=0, atol=1e-14)
    np.testing.assert_allclose(ST[0, 0], S1, rtol=0, atol=1e-14)
    np.testing.assert_allclose(RT[0, 0], R1, rtol=0, atol=1e-14)


@pytest.mark.parametrize("variant", [RLA, RDN])
def test_T1_zero_state_q_equals_k(variant):
    """With S0 = R0 = 0, q = k and |k| = 1 the first output is gam^2 clip(v):
    gamma enters once in the R update and once in the read-out (Section 3.4)."""
    rng = np.random.default_rng(3)
    D = 7
    k = rng.standard_normal(D)
    k /= np.linalg.norm(k)
    v = rng.standard_normal(D) * 2
    one = lambda a: np.asarray(a, dtype=np.float64).reshape(1, 1, 1, -1)
    s = lambda a: np.asarray([[[a]]], dtype=np.float64)
    gm = 0.37
    o, _, _ = oracle.fwd(variant, one(k), one(k), one(v), s(-0.2), s(0.6), s(gm), 1.0)
    np.testing.assert_allclose(o[0, 0, 0], gm * gm * np.clip(v, -1, 1), atol=1e-15)


# ------------------------------------------- golden hand-worked example
def _load_golden(name):
    vals = {}
    with open(os.path.join(GOLDEN, name)) as f:
        for line in f:
            line = line.split("#", 1)[0].strip()
            if not line:
                continue
            key, rest = line.split("=", 1)
            vals[key.strip()] = np.array([float(t) for t in rest.split()])
    return vals


@pytest.mark.parametrize("variant,fname", [(RDN, "rdn_T2_d2_hand.txt"), (RLA, "rla_T2_d2_hand.txt")])
def test_golden_hand_worked(variant, fname):
    gv = _load_golden(fname)
    q = gv["q"].reshape(1, 2, 1, 2)
    k = gv["k"].reshape(1, 2, 1, 2)
    v = gv["v"].reshape(1, 2, 1, 2)
    g = np.log(gv["alpha"]).reshape(1, 2, 1)
    be = gv["beta"].reshape(1, 2, 1)
    gm = gv["gamma"].reshape(1, 2, 1)
    o, ST, RT = oracle.fwd(variant, q, k, v, g, be, gm, float(gv["c"][0]))
    np.testing.assert_allclose(o.reshape(-1), gv["o"], atol=1e-14)
    np.testing.assert_allclose(ST.reshape(-1), gv["ST"], atol=1e-14)
    np.testing.assert_allclose(RT.reshape(-1), gv["RT"], atol=1e-14)


# ------------------------ textbook base models, written in the paper's d_v x d_k orientation
def _textbook_base(variant, x):
    """Gated DeltaNet (Table 1 / Section 2.2) or scalar-gated linear attention
    (Section 3.2), states d_v x d_k as in the paper.  Returns the per-token
    states before each update (paper orientation), the outputs S_t q_t and the
    final state."""
    q, k, v, g, be = x["q"], x["k"], x["v"], x["g"], x["beta"]
    B, T, H, Dk = q.shape
    Dv = v.shape[-1]
    prev = np.zeros((B, T, H, Dv, Dk))
    out = np.zeros((B, T, H, Dv))
    fin = np.zeros((B, H, Dv, Dk))
    for b in range(B):
        for h in range(H):
            S = np.zeros((Dv, Dk)) if x["S0"] is None else x["S0"][b, h].T.copy()
            for t in range(T):
                prev[b, t, h] = S
                kt, vt, a, bt = k[b, t, h], v[b, t, h], np.exp(g[b, t, h]), be[b, t, h]
                if variant == RDN:
                    S = a * S @ (np.eye(Dk) - bt * np.outer(kt, kt)) + bt * np.outer(vt, kt)
                else:
                    S = a * S + bt * np.outer(vt, kt)
                out[b, t, h] = S @ q[b, t, h]
            fin[b, h] = S
    return prev, out, fin


@pytest.mark.parametrize("variant", [RLA, RDN])
def test_base_state_is_textbook_and_independent_of_aux(variant):
    """P2 (Section 3.4): S follows GDN (RDN) / scalar-gated LA (RLA) and does not
    depend on R0, gamma or c."""
    x = _inputs()
    _, _, fin = _textbook_base(variant, x)
    _, ST, _ = _fwd(variant, x)
    np.testing.assert_allclose(ST, np.swapaxes(fin, -1, -2), atol=1e-13)
    y = dict(x)
    y["gamma"] = x["gamma"] * 0.3
    y["R0"] = x["R0"] * -2.0
    _, ST2, _ = _fwd(variant, y, c=0.05)
    np.testing.assert_allclose(ST2, ST, atol=1e-13)


@pytest.mark.parametrize("variant", [RLA, RDN])
def test_gamma_zero_reduces_to_base_model(variant):
    """P3 (Table 1): with gamma = 0 the auxiliary state only decays and
    o_t = a_t S_{t-1} q_t = o_t^base - beta_t (k_t.q_t)(v_t - a_t S_{t-1} k_t)
    (the base model's output minus its single-token correction; for the
    additive base the correction is beta_t (k_t.q_t) v_t)."""
    x = _inputs()
    x["gamma"] = np.zeros_like(x["gamma"])
    prev, out, _ = _textbook_base(variant, x)
    o, _, RT = _fwd(variant, x)
    a = np.exp(x["g"])
    kq = np.einsum("bthd,bthd->bth", x["k"], x["q"])
    if variant == RDN:
        corr = x["v"] - a[..., None] * np.einsum("bthjd,bthd->bthj", prev, x["k"])
    else:
        corr = x["v"]
    np.testing.assert_allclose(o, out - (x["beta"] * kq)[..., None] * corr, atol=1e-13)
    decay = np.exp(x["g"].sum(axis=1))  # [B,H]
    np.testing.assert_allclose(RT, decay[:, :, None, None] * x["R0"], atol=1e-14)


@pytest.mark.parametrize("variant", [RLA, RDN])
def test_clip_zero_no_aux_state(variant):
    """P4 (Section 3.3): c = 0 forces r = 0; with R0 = 0 the auxiliary state
    stays 0 and o_t = a_t S_{t-1} q_t."""
    x = _inputs()
    x["R0"] = None
    o, _, RT = _fwd(variant, x, c=0.0)
    assert np.all(RT == 0.0)
    prev, _, _ = _textbook_base(variant, x)
    base = np.exp(x["g"])[..., None] * np.einsum("bthjd,bthd->bthj", prev, x["q"])
    np.testing.assert_allclose(o, base, atol=1e-13)


# ------------------------------------------------------- P5: chunked == recurrent
@pytest.mark.parametrize("variant,name", [(RLA, "rla"), (RDN, "rdn")])
@pytest.mark.parametrize("C", [1, 16, 32, 64])
def test_chunkwise_equals_recurrent(variant, name, C):
    x = _inputs(B=1, T=100, H=2, D=16, Dv=12)
    o, ST, RT = _fwd(variant, x, c=0.8)
    oc, STc, RTc = chunk_fwd(name, x["q"], x["k"], x["v"], x["g"], x["beta"], x["gamma"], 0.8,
                             x["S0"], x["R0"], C=C)
    np.testing.assert_allclose(oc, o, atol=1e-11)
    np.testing.assert_allclose(STc, ST, atol=1e-11)
    np.testing.assert_allclose(RTc, RT, atol=1e-11)


@pytest.mark.parametrize("variant", [RLA, RDN])
def test_value_columns_independent(variant):
    """Each value column j of S, R, r and o depends only on column j of v and
    of the initial states (the clip is elementwise): slicing d_v is exact."""
    x = _inputs(B=1, T=40, H=2, D=8, Dv=10)
    o, ST, RT = _fwd(variant, x)
    parts = []
    for sl in (slice(0, 3), slice(3, 10)):
        y = dict(x)
        y["v"] = x["v"][..., sl].copy()
        y["S0"] = x["S0"][..., sl].copy()
        y["R0"] = x["R0"][..., sl].copy()
        parts.append(_fwd(variant, y))
    np.testing.assert_allclose(np.concatenate([p[0] for p in parts], -1), o, atol=1e-14)
    np.testing.assert_allclose(np.concatenate([p[1] for p in parts], -1), ST, atol=1e-14)
    np.testing.assert_allclose(np.concatenate([p[2] for p in parts], -1), RT, atol=1e-14)


# --------------------------------------------------------- P6: brute force, T <= 8
def _brute(variant, x, c):
    """Unrolled products, no recurrence reuse: S_t = (F_t...F_1) S0 + sum_i
    (F_t...F_{i+1}) beta_i k_i v_i^T with F_s = a_s (I - beta_s k_s k_s^T)
    (a_s I for RLA), residuals from the unrolled S_{t-1}, and likewise for R."""
    q, k, v = x["q"][0, :, 0], x["k"][0, :, 0], x["v"][0, :, 0]
    a = np.exp(x["g"][0, :, 0])
    be, gm = x["beta"][0, :, 0], x["gamma"][0, :, 0]
    S0, R0 = x["S0"][0, 0], x["R0"][0, 0]
    T, D = k.shape

    def F(s, rate):
        if variant == RDN:
            return a[s] * (np.eye(D) - rate[s] * np.outer(k[s], k[s]))
        return a[s] * np.eye(D)

    def prod(lo, hi, rate):  # F_{hi-1} ... F_{lo}
        M = np.eye(D)
        for s in range(lo, hi):
            M = F(s, rate) @ M
        return M

    def S_after(t):  # S_t with t tokens consumed
        out = prod(0, t, be) @ S0
        for i in range(t):
            out = out + prod(i + 1, t, be) @ (be[i] * np.outer(k[i], v[i]))
        return out

    r = [np.clip(v[i] - S_after(i).T @ k[i], -c, c) for i in range(T)]

    def R_after(t):
        out = prod(0, t, gm) @ R0
        for i in range(t):
            out = out + prod(i + 1, t, gm) @ (gm[i] * np.outer(k[i], r[i]))
        return out

    o = np.stack([a[t] * S_after(t).T @ q[t] + gm[t] * R_after(t + 1).T @ q[t] for t in range(T)])
    return o, S_after(T), R_after(T)


@pytest.mark.parametrize("variant", [RLA, RDN])
@pytest.mark.parametrize("T", [1, 2, 5, 8])
def test_brute_force_unrolled(variant, T):
    x = _inputs(B=1, T=T, H=1, D=5, Dv=4, seed=T)
    x["v"] = x["v"] * 2.0  # make the clip active
    o, ST, RT = _fwd(variant, x, c=0.9)
    ob, Sb, Rb = _brute(variant, x, 0.9)
    np.testing.assert_allclose(o[0, :, 0], ob, atol=1e-13)
    np.testing.assert_allclose(ST[0, 0], Sb, atol=1e-13)
    np.testing.assert_allclose(RT[0, 0], Rb, atol=1e-13)


# ---------------------------- P7: Appendix D pseudo-code semantics (own restatement)
def _listing_semantics_rla(q, k, v, alpha, beta, gamma):
    """What the Appendix D pseudo-code computes, restated: one head, zero
    initial states, states d_k x d_v, q and k L2-normalised inside the loop,
    residual clipped to [-1, 1], R updated before the read-out, S after it."""
    T, D = q.shape
    S = torch.zeros(D, D, dtype=torch.float64)
    R = torch.zeros(D, D, dtype=torch.float64)
    outs = []
    for t in range(T):
        qn = q[t] / q[t].norm()
        kn = k[t] / k[t].norm()
        resid = (v[t] - kn @ S).clamp(-1.0, 1.0)
        R = alpha[t] * R + gamma[t] * torch.outer(kn, resid)
        outs.append(alpha[t] * (qn @ S) + gamma[t] * (qn @ R))
        S = alpha[t] * S + beta[t] * torch.outer(kn, v[t])
    return torch.stack(outs)


def _listing_semantics_sgla(q, k, v, alpha, beta):
    """Appendix D baseline: scalar-gated LA, read-out after the update."""
    T, D = q.shape
    S = torch.zeros(D, D, dtype=torch.float64)
    outs = []
    for t in range(T):
        S = alpha[t] * S + beta[t] * torch.outer(k[t], v[t])
        outs.append(q[t] @ S)
    return torch.stack(outs)


def test_appendix_d_semantics():
    gen = torch.Generator().manual_seed(11)
    T, D = 30, 8
    q = torch.randn(T, D, generator=gen, dtype=torch.float64) * 3
    k = torch.randn(T, D, generator=gen, dtype=torch.float64) * 3
    v = torch.randn(T, D, generator=gen, dtype=torch.float64) * 2
    alpha = torch.sigmoid(torch.randn(T, generator=gen, dtype=torch.float64) + 2)
    beta = torch.sigmoid(torch.randn(T, generator=gen, dtype=torch.float64))
    gamma = torch.sigmoid(torch.randn(T, generator=gen, dtype=torch.float64))
    ref = _listing_semantics_rla(q, k, v, alpha, beta, gamma).numpy()
    qn = (q / q.norm(dim=-1, keepdim=True)).numpy()
    kn = (k / k.norm(dim=-1, keepdim=True)).numpy()
    sh = lambda a: a.numpy().reshape(1, T, 1, -1)
    o, _, _ = oracle.rla_fwd(qn.reshape(1, T, 1, D), kn.reshape(1, T, 1, D), sh(v),
                             np.log(alpha.numpy()).reshape(1, T, 1), beta.numpy().reshape(1, T, 1),
                             gamma.numpy().reshape(1, T, 1), 1.0)
    np.testing.assert_allclose(o[0, :, 0], ref, atol=1e-13)
    # the baseline sGLA (read-out after the update) equals RLA with gamma = 0
    # plus the current-token term beta_t (k_t.q_t) v_t (Table 1)
    sg = _listing_semantics_sgla(torch.from_numpy(qn), torch.from_numpy(kn), v, alpha, beta).numpy()
    o0, _, _ = oracle.rla_fwd(qn.reshape(1, T, 1, D), kn.reshape(1, T, 1, D), sh(v),
                              np.log(alpha.numpy()).reshape(1, T, 1), beta.numpy().reshape(1, T, 1),
                              np.zeros((1, T, 1)), 1.0)
    kq = (qn * kn).sum(-1)
    np.testing.assert_allclose(o0[0, :, 0] + (beta.numpy() * kq)[:, None] * v.numpy(), sg,
                               atol=1e-13)


# ------------------------------------------------------------- P8: linearity
def test_rla_linear_in_v_without_clip():
    """RLA with c = inf and zero initial states is linear in v (every update is
    additive); a finite c breaks linearity (Section 3.3)."""
    x = _inputs(nonzero=False)
    y = dict(x)
    y["v"] = _inputs(nonzero=False, seed=5)["v"]
    z = dict(x)
    z["v"] = x["v"] + 2.5 * y["v"]
    lin = lambda c: (_fwd(RLA, z, c)[0], _fwd(RLA, x, c)[0] + 2.5 * _fwd(RLA, y, c)[0])
    a, b = lin(np.inf)
    np.testing.assert_allclose(a, b, atol=1e-12)
    a, b = lin(0.3)
    assert np.abs(a - b).max() > 1e-2


# ------------------------------------------------------------- P9: gradients
def _torch_recurrence(variant, q, k, v, alpha, beta, gamma, c, S0, R0):
    """Independent autograd-able restatement in the paper's d_v x d_k
    orientation, vectorised over (b, h)."""
    B, T, H, Dk = q.shape
    S, R = S0.transpose(-1, -2), R0.transpose(-1, -2)  # [B,H,Dv,Dk]
    outs = []
    eye = torch.eye(Dk, dtype=q.dtype)
    for t in range(T):
        qt, kt, vt = q[:, t], k[:, t], v[:, t]  # [B,H,D]
        a, bt, gt = alpha[:, t, :, None, None], beta[:, t, :, None, None], gamma[:, t, :, None, None]
        kkT = kt[..., :, None] * kt[..., None, :]
        r = torch.clamp(vt - (S @ kt[..., None])[..., 0], -c, c)
        if variant == RDN:
            Rn = a * R @ (eye - gt * kkT) + gt * r[..., :, None] * kt[..., None, :]
            Sn = a * S @ (eye - bt * kkT) + bt * vt[..., :, None] * kt[..., None, :]
        else:
            Rn = a * R + gt * r[..., :, None] * kt[..., None, :]
            Sn = a * S + bt * vt[..., :, None] * kt[..., None, :]
        outs.append(a[..., 0] * (S @ qt[..., None])[..., 0] + gt[..., 0] * (Rn @ qt[..., None])[..., 0])
        S, R = Sn, Rn
    return torch.stack(outs, 1), S.transpose(-1, -2), R.transpose(-1, -2)


@pytest.mark.parametrize("variant", [RLA, RDN])
def test_backward_matches_autograd(variant):
    x = _inputs(B=2, T=70, H=2, D=6, Dv=5)  # T > 64: crosses an oracle checkpoint
    x["v"] = x["v"] * 1.5
    c = 0.8
    dST = np.random.default_rng(1).standard_normal(x["S0"].shape)
    dRT = np.random.default_rng(2).standard_normal(x["R0"].shape)
    T_ = {n: torch.tensor(a, requires_grad=True) for n, a in x.items() if a is not None and n != "dO"}
    alpha = torch.exp(T_["g"])
    o, ST, RT = _torch_recurrence(variant, T_["q"], T_["k"], T_["v"], alpha, T_["beta"],
                                  T_["gamma"], c, T_["S0"], T_["R0"])
    loss = (o * torch.from_numpy(x["dO"])).sum() + (ST * torch.from_numpy(dST)).sum() \
        + (RT * torch.from_numpy(dRT)).sum()
    loss.backward()
    d = oracle.bwd(variant, x["q"], x["k"], x["v"], x["g"], x["beta"], x["gamma"], c,
                   x["S0"], x["R0"], x["dO"], dST, dRT)
    for name, key in [("dq", "q"), ("dk", "k"), ("dv", "v"), ("dg", "g"), ("dbeta", "beta"),
                      ("dgamma", "gamma"), ("dS0", "S0"), ("dR0", "R0")]:
        np.testing.assert_allclose(d[name], T_[key].grad.numpy(), atol=1e-11, err_msg=name)


def test_backward_alpha_chain_rule():
    """dg = alpha * dL/dalpha: check against autograd taken w.r.t. alpha."""
    x = _inputs(B=1, T=12, H=1, D=4)
    c = 1.0
    alpha = torch.tensor(np.exp(x["g"]), requires_grad=True)
    t = {n: torch.tensor(a) for n, a in x.items() if a is not None}
    o, _, _ = _torch_recurrence(RDN, t["q"], t["k"], t["v"], alpha, t["beta"], t["gamma"], c,
                                t["S0"], t["R0"])
    (o * t["dO"]).sum().backward()
    d = oracle.rdn_bwd(x["q"], x["k"], x["v"], x["g"], x["beta"], x["gamma"], c, x["S0"],
                       x["R0"], x["dO"])
    np.testing.assert_allclose(d["dg"] / np.exp(x["g"]), alpha.grad.numpy(), atol=1e-12)


@pytest.mark.parametrize("variant", [RLA, RDN])
def test_backward_finite_differences(variant):
    """Central differences of the oracle's own forward on a few coordinates of
    every input (clip active, but no element near the threshold)."""
    x = _inputs(B=1, T=9, H=1, D=4, Dv=3, seed=4)
    c = 0.9
    x["v"], n = oracle.clip_margin_condition(variant, x["q"], x["k"], x["v"], x["g"], x["beta"],
                                             x["gamma"], c, x["S0"], x["R0"], margin=1e-3,
                                             quant="f64")
    d = oracle.bwd(variant, x["q"], x["k"], x["v"], x["g"], x["beta"], x["gamma"], c, x["S0"],
                   x["R0"], x["dO"])

    def loss(y):
        o, _, _ = _fwd(variant, y, c)
        return float((o * x["dO"]).sum())

    rng = np.random.default_rng(0)
    eps = 1e-6
    for key, gname in [("q", "dq"), ("k", "dk"), ("v", "dv"), ("g", "dg"), ("beta", "dbeta"),
                       ("gamma", "dgamma"), ("S0", "dS0"), ("R0", "dR0")]:
        for _ in range(3):
            idx = tuple(rng.integers(0, s) for s in x[key].shape)
            yp, ym = dict(x), dict(x)
            yp[key] = x[key].copy()
            ym[key] = x[key].copy()
            yp[key][idx] += eps
            ym[key][idx] -= eps
            fd = (loss(yp) - loss(ym)) / (2 * eps)
            assert abs(fd - d[gname][idx]) < 1e-6 * max(1.0, abs(fd)), (key, idx, fd, d[gname][idx])


def test_clip_tie_passes_gradient():
    """Reading of Section 3.3: at |v - S_{t-1}k| == c exactly the clip's
    derivative is taken as 1 (inclusive mask)."""
    D = 2
    one = lambda a: np.asarray(a, dtype=np.float64).reshape(1, 1, 1, -1)
    s = lambda a: np.asarray([[[a]]], dtype=np.float64)
    k = one([1.0, 0.0])
    q = one([1.0, 0.0])
    v = one([0.5, 0.75])  # S0 = 0: x = v, first element exactly at c = 0.5
    dO = one([1.0, 1.0])
    gm = 0.5
    d = oracle.rdn_bwd(q, k, v, s(-0.1), s(0.4), s(gm), 0.5, None, None, dO)
    # o = gam^2 (k.q) clip(v) + a S0 q ... -> d o_j / d v_j = gam^2 on |v_j| <= c
    np.testing.assert_allclose(d["dv"][0, 0, 0, 0], gm * gm + 0.4 * 0.0 * 1, atol=1e-15)
    assert d["dv"][0, 0, 0, 1] == pytest.approx(0.0, abs=1e-15)


def test_margin_conditioning():
    """After conditioning, every fp64 residual is at least `margin` from c and
    the moved values are representable in the stated dtype."""
    x = _inputs(B=1, T=50, H=2, D=8, nonzero=False)
    x["v"] = x["v"].astype(np.float32).astype(np.float64)
    c, m = 0.6, 5e-3
    v2, n = oracle.clip_margin_condition(RDN, x["q"], x["k"], x["v"], x["g"], x["beta"],
                                         x["gamma"], c, margin=m, quant="bf16")
    assert n > 0
    y = dict(x)
    y["v"] = v2
    _, _, _, r = _fwd(RDN, y, c, return_residual=True)
    o, ST, RT = _fwd(RDN, y, c)
    # recompute x = v - p token by token via the residual: |x| - c margin holds
    # wherever the residual is not clipped (|r| < c) and where it is (|r| == c)
    moved = v2 != x["v"]
    assert np.all(v2[moved].astype(np.float32) == v2[moved])  # fp32-exact
    bf = torch.tensor(v2[moved]).to(torch.bfloat16).double().numpy()
    np.testing.assert_array_equal(bf, v2[moved])
    inside = np.abs(r) < c
    assert np.all(np.abs(np.abs(r[inside]) - c) >= m - 1e-12)


def test_decode_step_chain_equals_forward():
    """T successive single-token steps reproduce the sequence forward (P10)."""
    x = _inputs(B=3, T=6, H=2, D=5)
    for variant in (RLA, RDN):
        o, ST, RT = _fwd(variant, x)
        S, R = x["S0"].copy(), x["R0"].copy()
        for t in range(6):
            ot, S, R = oracle.decode_step(variant, x["q"][:, t], x["k"][:, t], x["v"][:, t],
                                          x["g"][:, t], x["beta"][:, t], x["gamma"][:, t], 1.0, S, R)
            np.testing.assert_allclose(ot, o[:, t], atol=1e-14)
        np.testing.assert_allclose(S, ST, atol=1e-14)
        np.testing.assert_allclose(R, RT, atol=1e-14)


def test_split_sequence_continuation():
    """fwd(T1) -> (S, R) -> fwd(T2, S0=S, R0=R) equals fwd(T1 + T2): the
    final states are the layer's resume point."""
    x = _inputs(B=1, T=40, H=2, D=6)
    o, ST, RT = _fwd(RDN, x)
    a = {n: (v[:, :17] if v is not None and v.ndim >= 3 and v.shape[1] == 40 else v)
         for n, v in x.items()}
    b = {n: (v[:, 17:] if v is not None and v.ndim >= 3 and v.shape[1] == 40 else v)
         for n, v in x.items()}
    oa, Sa, Ra = _fwd(RDN, a)
    b["S0"], b["R0"] = Sa, Ra
    ob, Sb, Rb = _fwd(RDN, b)
    np.testing.assert_allclose(np.concatenate([oa, ob], 1), o, atol=1e-13)
    np.testing.assert_allclose(Sb, ST, atol=1e-13)
    np.testing.assert_allclose(Rb, RT, atol=1e-13)


@pytest.mark.parametrize("variant,name", [(RLA, "rla"), (RDN, "rdn")])
@pytest.mark.parametrize("C", [1, 16, 64])
def test_chunkwise_backward_equals_bptt(variant, name, C):
    """The reverse-mode chunk algebra (test helper) equals the oracle's
    back-propagation through time (and so, via the autograd pins, the exact
    gradient)."""
    from tests.chunk_algebra import chunk_bwd
    x = _inputs(B=1, T=100, H=2, D=8, Dv=6)
    x["v"] = x["v"] * 1.5
    c = 0.8
    dST = np.random.default_rng(1).standard_normal(x["S0"].shape)
    dRT = np.random.default_rng(2).standard_normal(x["R0"].shape)
    ref = oracle.bwd(variant, x["q"], x["k"], x["v"], x["g"], x["beta"], x["gamma"], c,
                     x["S0"], x["R0"], x["dO"], dST, dRT, scale=0.7)
    got = chunk_bwd(name, x["q"], x["k"], x["v"], x["g"], x["beta"], x["gamma"], c, x["S0"],
                    x["R0"], x["dO"], dST, dRT, C=C, scale=0.7)
    for key in ref:
        np.testing.assert_allclose(got[key], ref[key], atol=1e-10, err_msg=key)


# ------------------------------------------------ q, k prologue (SiLU, L2 norm)
def test_qk_prologue_rows_have_unit_norm_and_silu_direction():
    """Each row of the output is the unit vector along SiLU(x): norm 1, and
    parallel to x * sigmoid(x) computed with scipy's logistic function."""
    from scipy.special import expit
    x = np.random.default_rng(3).standard_normal((5, 7, 128)) * 2.0
    y = oracle.qk_prologue(x)
    np.testing.assert_allclose(np.linalg.norm(y, axis=-1), 1.0, atol=1e-14)
    u = x * expit(x)
    np.testing.assert_allclose(y * np.linalg.norm(u, axis=-1, keepdims=True), u, atol=1e-12)


def test_qk_prologue_closed_forms():
    """One-element rows: y = sign(SiLU(x)) (SiLU(x) > 0 iff x > 0); an all-zero
    row falls under the floor and stays zero; x = ln 3 has sigmoid 3/4."""
    x = np.array([[2.0], [-0.5], [0.0]])
    y = oracle.qk_prologue(x)
    np.testing.assert_array_equal(y[:, 0], [1.0, -1.0, 0.0])
    x2 = np.array([[np.log(3.0), 0.0]])  # SiLU = (ln 3) 3/4 and 0: the unit row (1, 0)
    np.testing.assert_allclose(oracle.qk_prologue(x2), [[1.0, 0.0]], atol=1e-15)
    # the norm floor: y = u / eps for rows whose SiLU is tiny
    tiny = np.array([[1e-14, -2e-14]])
    u = tiny / (1.0 + np.exp(-tiny))
    np.testing.assert_allclose(oracle.qk_prologue(tiny, eps=1e-12), u / 1e-12, rtol=1e-12)


def test_qk_prologue_backward_matches_autograd():
    """Against fp64 autograd of torch's silu and normalize (library routines)."""
    rng = np.random.default_rng(5)
    x = rng.standard_normal((3, 4, 64)) * 1.5
    dy = rng.standard_normal(x.shape)
    t = torch.tensor(x, requires_grad=True)
    y = torch.nn.functional.normalize(torch.nn.functional.silu(t), dim=-1, eps=1e-12)
    (y * torch.from_numpy(dy)).sum().backward()
    np.testing.assert_allclose(oracle.qk_prologue(x), y.detach().numpy(), atol=1e-14)
    np.testing.assert_allclose(oracle.qk_prologue_bwd(x, dy), t.grad.numpy(), atol=1e-12)


def test_qk_prologue_backward_finite_differences():
    rng = np.random.default_rng(6)
    x = rng.standard_normal((2, 16))
    dy = rng.standard_normal(x.shape)
    g = oracle.qk_prologue_bwd(x, dy)
    eps = 1e-6
    for idx in [(0, 0), (0, 7), (1, 3), (1, 15)]:
        xp, xm = x.copy(), x.copy()
        xp[idx] += eps
        xm[idx] -= eps
        fd = ((oracle.qk_prologue(xp) - oracle.qk_prologue(xm)) * dy).sum() / (2 * eps)
        assert abs(fd - g[idx]) < 1e-7, (idx, fd, g[idx])


@pytest.mark.parametrize("variant", [RLA, RDN])
def test_tied_gate_gradient_matches_autograd(variant):
    """Tied gates (gamma = beta, the paper's tied-gate ablation): the gradient
    w.r.t. the shared gate, formed from the oracle as dbeta + dgamma of the
    untied computation at gamma = beta, equals fp64 autograd of the recurrence
    driven by one gate tensor."""
    x = _inputs(B=1, T=40, H=2, D=5, Dv=4, seed=8)
    c = 0.7
    T_ = {n: torch.tensor(a, requires_grad=True) for n, a in x.items() if a is not None and n != "dO"}
    o, ST, RT = _torch_recurrence(variant, T_["q"], T_["k"], T_["v"], torch.exp(T_["g"]),
                                  T_["beta"], T_["beta"], c, T_["S0"], T_["R0"])
    (o * torch.from_numpy(x["dO"])).sum().backward()
    d = oracle.bwd(variant, x["q"], x["k"], x["v"], x["g"], x["beta"], x["beta"], c, x["S0"],
                   x["R0"], x["dO"])
    np.testing.assert_allclose(d["dbeta"] + d["dgamma"], T_["beta"].grad.numpy(), atol=1e-11)


def test_qk_round_margin_condition():
    """The prologue-rounding conditioner: its rows are bf16 values, every fp64
    y lands at least the margin away from a bf16 rounding tie, rows that were
    clear are untouched, and y computed in fp32 (the library's precision,
    with a plain sum of squares) then rounds to bf16 exactly like the fp64 y."""
    import torch
    rng = np.random.default_rng(3)
    x = torch.from_numpy(rng.standard_normal((4096, 128))).to(torch.bfloat16).double().numpy()
    x[7] = 0.0  # a row under the floor stays as it is (y = 0)
    xc, moved = oracle.qk_round_margin_condition(x)
    assert moved > 0
    assert np.array_equal(torch.from_numpy(xc).to(torch.bfloat16).double().numpy(), xc)
    y0 = oracle.qk_prologue(x)
    clear = (oracle._bf16_tie_distance(y0) >= 2.0 ** -9).all(-1)
    assert np.array_equal(xc[clear], x[clear]) and not clear.all()
    y = oracle.qk_prologue(xc)
    assert oracle._bf16_tie_distance(y).min() >= 2.0 ** -9
    x32 = xc.astype(np.float32)
    u32 = x32 / (np.float32(1.0) + np.exp(-x32))
    y32 = u32 / np.maximum(np.sqrt((u32 * u32).sum(-1, keepdims=True, dtype=np.float32)),
                           np.float32(1e-12))
    assert torch.equal(torch.from_numpy(y).to(torch.bfloat16),
                       torch.from_numpy(y32.astype(np.float64)).to(torch.bfloat16))
    # the tie distance itself: a bf16 value is 1/2 from a tie, a midpoint 0
    assert oracle._bf16_tie_distance(np.array([1.0, 1.0 + 2.0 ** -8, 3.0]))[[0, 2]].min() == 0.5
    assert oracle._bf16_tie_distance(np.array([1.0 + 2.0 ** -8]))[0] == 0.0
