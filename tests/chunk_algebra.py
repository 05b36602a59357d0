"""Chunkwise-parallel form of RLA / RDN, restated in fp64 numpy.

Test helper only (not the oracle, not the CUDA path).  It writes out the
chunk algebra that the CUDA kernels implement, so that the tests can check
it against the token recurrence (Section 3.4) independently of any GPU.

Within a chunk of C tokens starting from states S0, R0 ([d_k][d_v] storage),
with b_t = sum_{s<=t} g_s (in-chunk cumulative log-decay, b_0 = 0) and
Gam_t = exp(b_t):

  delta rule written as S_t = a_t S_{t-1} + beta_t k_t e_t^T with the
  delta error e_t = v_t - a_t S_{t-1}^T k_t  (Section 2.2 / 3.4), so
      S_t = Gam_t S0 + sum_{i<=t} (Gam_t/Gam_i) beta_i k_i e_i^T.
  Stacking e_t gives (I + A) E = V - diag(Gam) K S0 with
      A[t,i] = exp(b_t - b_i) beta_i (k_t . k_i), i < t      (WY / UT form)
  hence E = T (V - diag(Gam) K S0), T = (I + A)^-1.
  RLA has no delta term: E = V.

  residual prediction (undecayed, Section 3.3):
      P_t = S_{t-1}^T k_t = exp(b_{t-1}) (K S0)_t
            + sum_{i<t} exp(b_{t-1} - b_i) beta_i (k_t . k_i) e_i
  base output a_t S_{t-1}^T q_t = Gam_t (Q S0)_t
            + sum_{i<t} exp(b_t - b_i) beta_i (q_t . k_i) e_i
  chunk-end state  S_C = Gam_C S0 + K^T diag(beta_i exp(b_C - b_i)) E

  the auxiliary pass is the same algebra with values clip(V - P), rate gamma
  and state R; its read-out R_t^T q_t includes token t:
      Gam_t (Q R0)_t + sum_{i<=t} exp(b_t - b_i) gamma_i (q_t . k_i) e2_i
  output o_t = base_t + gamma_t * (R_t^T q_t).
"""
from __future__ import annotations

import numpy as np


def chunk_fwd(variant, q, k, v, g, beta, gamma, c, S0=None, R0=None, C=64, scale=1.0):
    """variant: "rla" | "rdn".  Arrays as in the oracle (float64)."""
    q, k, v, g, beta, gamma = (np.asarray(x, dtype=np.float64) for x in (q, k, v, g, beta, gamma))
    B, T, H, Dk = q.shape
    Dv = v.shape[-1]
    o = np.zeros((B, T, H, Dv))
    ST = np.zeros((B, H, Dk, Dv))
    RT = np.zeros((B, H, Dk, Dv))
    for b in range(B):
        for h in range(H):
            S = np.zeros((Dk, Dv)) if S0 is None else np.array(S0[b, h], dtype=np.float64)
            R = np.zeros((Dk, Dv)) if R0 is None else np.array(R0[b, h], dtype=np.float64)
            for t0 in range(0, T, C):
                t1 = min(t0 + C, T)
                n = t1 - t0
                K = k[b, t0:t1, h]
                Q = q[b, t0:t1, h] * scale
                V = v[b, t0:t1, h]
                gc, bc, gm = g[b, t0:t1, h], beta[b, t0:t1, h], gamma[b, t0:t1, h]
                cum = np.cumsum(gc)
                cum_prev = cum - gc
                Gam = np.exp(cum)
                Gam_prev = np.exp(cum_prev)
                strict = np.tril(np.ones((n, n), dtype=bool), -1)
                incl = np.tril(np.ones((n, n), dtype=bool), 0)
                diff = cum[:, None] - cum[None, :]
                dec = np.where(incl, np.exp(np.where(incl, diff, 0.0)), 0.0)
                diff_prev = cum_prev[:, None] - cum[None, :]
                dec_prev = np.where(strict, np.exp(np.where(strict, diff_prev, 0.0)), 0.0)
                KK = K @ K.T
                QK = Q @ K.T
                KS = K @ S
                QS = Q @ S
                if variant == "rdn":
                    A = np.where(strict, dec * KK, 0.0) * bc[None, :]
                    Tm = np.linalg.inv(np.eye(n) + A)
                    E = Tm @ (V - Gam[:, None] * KS)
                else:
                    E = V
                Ap = dec_prev * KK * bc[None, :]
                P = Gam_prev[:, None] * KS + Ap @ E
                Mq = np.where(strict, dec * QK, 0.0) * bc[None, :]
                Ob = Gam[:, None] * QS + Mq @ E
                wS = bc * np.exp(cum[-1] - cum)
                S_new = Gam[-1] * S + K.T @ (wS[:, None] * E)

                Rv = np.clip(V - P, -c, c)
                KR = K @ R
                QR = Q @ R
                if variant == "rdn":
                    Ag = np.where(strict, dec * KK, 0.0) * gm[None, :]
                    Tg = np.linalg.inv(np.eye(n) + Ag)
                    E2 = Tg @ (Rv - Gam[:, None] * KR)
                else:
                    E2 = Rv
                M2 = dec * QK * gm[None, :]
                Oa = Gam[:, None] * QR + M2 @ E2
                o[b, t0:t1, h] = Ob + gm[:, None] * Oa
                wR = gm * np.exp(cum[-1] - cum)
                R = Gam[-1] * R + K.T @ (wR[:, None] * E2)
                S = S_new
            ST[b, h] = S
            RT[b, h] = R
    return o, ST, RT


def _pieces(variant, K, Q, V, gc, bc, gm, S0, R0, c):
    """Forward intermediates of one chunk (see the module docstring)."""
    n = K.shape[0]
    f = {}
    cum = np.cumsum(gc)
    cprev = cum - gc
    strict = np.tril(np.ones((n, n), dtype=bool), -1)
    incl = np.tril(np.ones((n, n), dtype=bool), 0)
    dec = np.where(incl, np.exp(np.where(incl, cum[:, None] - cum[None, :], 0.0)), 0.0)
    decp = np.where(strict, np.exp(np.where(strict, cprev[:, None] - cum[None, :], 0.0)), 0.0)
    f.update(cum=cum, cprev=cprev, Gam=np.exp(cum), Gprev=np.exp(cprev), GamC=np.exp(cum[-1]),
             dec=dec, decp=decp, strict=strict, incl=incl)
    KK, QK = K @ K.T, Q @ K.T
    f.update(KK=KK, QK=QK, KS=K @ S0, QS=Q @ S0, KR=K @ R0, QR=Q @ R0)
    if variant == "rdn":
        f["Ab"] = np.where(strict, dec * KK, 0.0) * bc[None, :]
        f["Tb"] = np.linalg.inv(np.eye(n) + f["Ab"])
        f["X"] = V - f["Gam"][:, None] * f["KS"]
        f["E"] = f["Tb"] @ f["X"]
    else:
        f["E"] = V
    f["Ap"] = decp * KK * bc[None, :]
    f["P"] = f["Gprev"][:, None] * f["KS"] + f["Ap"] @ f["E"]
    f["Mq"] = np.where(strict, dec * QK, 0.0) * bc[None, :]
    f["Ob"] = f["Gam"][:, None] * f["QS"] + f["Mq"] @ f["E"]
    f["wS"] = bc * np.exp(cum[-1] - cum)
    f["xres"] = V - f["P"]
    f["Rv"] = np.clip(f["xres"], -c, c)
    f["mask"] = np.abs(f["xres"]) <= c
    if variant == "rdn":
        f["Ag"] = np.where(strict, dec * KK, 0.0) * gm[None, :]
        f["Tg"] = np.linalg.inv(np.eye(n) + f["Ag"])
        f["X2"] = f["Rv"] - f["Gam"][:, None] * f["KR"]
        f["E2"] = f["Tg"] @ f["X2"]
    else:
        f["E2"] = f["Rv"]
    f["M2"] = dec * QK * gm[None, :]
    f["Oa"] = f["Gam"][:, None] * f["QR"] + f["M2"] @ f["E2"]
    f["wR"] = gm * np.exp(cum[-1] - cum)
    f["SC"] = f["GamC"] * S0 + K.T @ (f["wS"][:, None] * f["E"])
    f["RC"] = f["GamC"] * R0 + K.T @ (f["wR"][:, None] * f["E2"])
    return f


def _chunk_adjoint(variant, K, Q, V, gc, bc, gm, S0, R0, f, dO, dSC, dRC):
    """Reverse mode of one chunk.  Returns (dK, dQ, dV, dg, dbeta, dgamma,
    dS0, dR0); dQ is w.r.t. the scaled Q."""
    n = K.shape[0]
    strict, incl = f["strict"], f["incl"]
    Gam, Gprev = f["Gam"], f["Gprev"]
    # ---- auxiliary (R) pass
    dgam = np.sum(dO * f["Oa"], 1)
    dOa = gm[:, None] * dO
    dGam = np.sum(dOa * f["QR"], 1)
    dQR = Gam[:, None] * dOa
    dM2 = np.where(incl, dOa @ f["E2"].T, 0.0)
    dE2 = f["M2"].T @ dOa
    dR0 = f["GamC"] * dRC
    dGamC = np.sum(dRC * R0)
    KdR = K @ dRC
    dE2 += f["wR"][:, None] * KdR
    dwR = np.sum(KdR * f["E2"], 1)
    dK = (f["wR"][:, None] * f["E2"]) @ dRC.T
    if variant == "rdn":
        dX2 = f["Tg"].T @ dE2
        dAg = np.where(strict, -(dX2 @ f["E2"].T), 0.0)
        dRv = dX2
        dKR = -Gam[:, None] * dX2
        dGam -= np.sum(dX2 * f["KR"], 1)
    else:
        dAg = np.zeros((n, n))
        dRv = dE2
        dKR = np.zeros_like(dE2)
    dR0 += K.T @ dKR + Q.T @ dQR
    dK += dKR @ R0.T
    dQ = dQR @ R0.T
    # ---- clip
    dV = dRv * f["mask"]
    dP = -dV
    # ---- base (S) pass
    dGam += np.sum(dO * f["QS"], 1)
    dQS = Gam[:, None] * dO
    dMq = np.where(strict, dO @ f["E"].T, 0.0)
    dE = f["Mq"].T @ dO
    dGprev = np.sum(dP * f["KS"], 1)
    dKS = Gprev[:, None] * dP
    dAp = np.where(strict, dP @ f["E"].T, 0.0)
    dE += f["Ap"].T @ dP
    dS0 = f["GamC"] * dSC
    dGamC += np.sum(dSC * S0)
    KdS = K @ dSC
    dE += f["wS"][:, None] * KdS
    dwS = np.sum(KdS * f["E"], 1)
    dK += (f["wS"][:, None] * f["E"]) @ dSC.T
    if variant == "rdn":
        dX = f["Tb"].T @ dE
        dAb = np.where(strict, -(dX @ f["E"].T), 0.0)
        dV += dX
        dKS -= Gam[:, None] * dX
        dGam -= np.sum(dX * f["KS"], 1)
    else:
        dAb = np.zeros((n, n))
        dV += dE
    dS0 += K.T @ dKS + Q.T @ dQS
    dK += dKS @ S0.T
    dQ += dQS @ S0.T
    # ---- C x C matrices -> Gram matrices, rates and cumulative log-decay
    dcum = np.zeros(n)
    dcprev = np.zeros(n)
    dbeta = np.zeros(n)
    dKK = np.zeros((n, n))
    dQK = np.zeros((n, n))
    for dM, M, base, rate, which, prev in ((dAp, f["Ap"], f["KK"], bc, "b", True),
                                           (dMq, f["Mq"], f["QK"], bc, "b", False),
                                           (dM2, f["M2"], f["QK"], gm, "g", False),
                                           (dAb, f.get("Ab"), f["KK"], bc, "b", False),
                                           (dAg, f.get("Ag"), f["KK"], gm, "g", False)):
        if M is None:
            continue
        G = dM * M
        if prev:
            dcprev += G.sum(1)
            d = f["decp"]
        else:
            dcum += G.sum(1)
            d = f["dec"]
        dcum -= G.sum(0)
        drate = np.sum(dM * d * base, 0)
        if which == "b":
            dbeta += drate
        else:
            dgam += drate
        contrib = dM * d * rate[None, :]
        if base is f["KK"]:
            dKK += contrib
        else:
            dQK += contrib
    eC = np.exp(f["cum"][-1] - f["cum"])
    dbeta += dwS * eC
    dgam += dwR * eC
    dcum[-1] += np.sum(dwS * f["wS"]) + np.sum(dwR * f["wR"]) + dGamC * f["GamC"]
    dcum -= dwS * f["wS"] + dwR * f["wR"]
    dcum += dGam * Gam
    dcprev += dGprev * Gprev
    dK += (dKK + dKK.T) @ K + dQK.T @ Q
    dQ += dQK @ K
    # cum_t = sum_{s<=t} g_s ; cprev_t = sum_{s<t} g_s
    dg = np.cumsum(dcum[::-1])[::-1] + (np.cumsum(dcprev[::-1])[::-1] - dcprev)
    return dK, dQ, dV, dg, dbeta, dgam, dS0, dR0


def chunk_bwd(variant, q, k, v, g, beta, gamma, c, S0, R0, dO, dST=None, dRT=None, C=64,
              scale=1.0):
    """Chunkwise backward (reverse scan over chunks carrying dS, dR)."""
    q, k, v, g, beta, gamma, dO = (np.asarray(x, dtype=np.float64)
                                   for x in (q, k, v, g, beta, gamma, dO))
    B, T, H, Dk = q.shape
    Dv = v.shape[-1]
    out = dict(dq=np.zeros_like(q), dk=np.zeros_like(k), dv=np.zeros_like(v),
               dg=np.zeros_like(g), dbeta=np.zeros_like(beta), dgamma=np.zeros_like(gamma),
               dS0=np.zeros((B, H, Dk, Dv)), dR0=np.zeros((B, H, Dk, Dv)))
    for b in range(B):
        for h in range(H):
            S = np.zeros((Dk, Dv)) if S0 is None else np.array(S0[b, h], dtype=np.float64)
            R = np.zeros((Dk, Dv)) if R0 is None else np.array(R0[b, h], dtype=np.float64)
            starts, states = list(range(0, T, C)), []
            for t0 in starts:  # chunk-start states (the forward's checkpoints)
                t1 = min(t0 + C, T)
                states.append((S, R))
                f = _pieces(variant, k[b, t0:t1, h], q[b, t0:t1, h] * scale, v[b, t0:t1, h],
                            g[b, t0:t1, h], beta[b, t0:t1, h], gamma[b, t0:t1, h], S, R, c)
                S, R = f["SC"], f["RC"]
            dS = np.zeros((Dk, Dv)) if dST is None else np.array(dST[b, h], dtype=np.float64)
            dR = np.zeros((Dk, Dv)) if dRT is None else np.array(dRT[b, h], dtype=np.float64)
            for t0, (Sc, Rc) in reversed(list(zip(starts, states))):
                t1 = min(t0 + C, T)
                K, Q, V = k[b, t0:t1, h], q[b, t0:t1, h] * scale, v[b, t0:t1, h]
                gc, bc, gm = g[b, t0:t1, h], beta[b, t0:t1, h], gamma[b, t0:t1, h]
                f = _pieces(variant, K, Q, V, gc, bc, gm, Sc, Rc, c)
                dK, dQ, dV, dgc, dbc, dgm, dS, dR = _chunk_adjoint(
                    variant, K, Q, V, gc, bc, gm, Sc, Rc, f, dO[b, t0:t1, h], dS, dR)
                out["dk"][b, t0:t1, h] = dK
                out["dq"][b, t0:t1, h] = dQ * scale
                out["dv"][b, t0:t1, h] = dV
                out["dg"][b, t0:t1, h] = dgc
                out["dbeta"][b, t0:t1, h] = dbc
                out["dgamma"][b, t0:t1, h] = dgm
            out["dS0"][b, h] = dS
            out["dR0"][b, h] = dR
    return out
