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
