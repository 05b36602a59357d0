"""Pins for the oracle's variants of the method (oracle.fwd / bwd `mods`),
checked against what the paper and mathematics fix (CPU only).

  DECAYED    residual against the decayed prediction a_t S_{t-1} k_t, the
             gated-delta error (Table 1 of Section 2.3, Section 3.4)
  PLAIN      ungated combine o_t = S_{t-1} q_t + R_t q_t (Section 4.3, output
             combination ablation)
  TANH       log-cosh residual c tanh(x / c) (Appendix B)
  STATELESS  R_t = r_t k_t^T, no accumulated auxiliary state (Section 4.3,
             residual-fitting ablation)

The pins use special cases where a variant must coincide with something
computed another way: the base-model state path (pinned on its own in
test_oracle_pins.py) run on prefixes of the sequence, a loss whose gradient
the paper names, or a limit where two variants are the same map.
"""
import numpy as np
import pytest

import oracle
from oracle import DECAYED, PLAIN, RDN, RLA, STATELESS, TANH
from rdn_synthetic import make_inputs


def _inputs(B=1, T=11, H=2, D=6, Dv=5, seed=0, state_std=0.3):
    x = make_inputs(B, T, H, D, dtype="f32", nonzero_state=True, with_grad_out=True, seed=seed,
                    Dv=Dv, state_std=state_std)
    return {n: (None if t is None else t.double().numpy()) for n, t in x.items()}


def _fwd(variant, x, c=1.0, mods=0, **kw):
    return oracle.fwd(variant, x["q"], x["k"], x["v"], x["g"], x["beta"], x["gamma"], c,
                      x["S0"], x["R0"], mods=mods, **kw)


def _prefix(x, t):
    """The inputs restricted to tokens [0, t)."""
    y = dict(x)
    for n in ("q", "k", "v", "g", "beta", "gamma", "dO"):
        y[n] = np.ascontiguousarray(x[n][:, :t])
    return y


# ------------------------------------------------------------ DECAYED, TANH
@pytest.mark.parametrize("variant", [RLA, RDN])
@pytest.mark.parametrize("mods", [DECAYED, TANH, DECAYED | TANH])
def test_residual_variants_from_the_base_path(variant, mods):
    """The residual variants change only what R fits: (i) r_t is the residual
    map of v_t - p_t with p_t = S_{t-1} k_t (DECAYED: a_t S_{t-1} k_t), S_{t-1}
    the base state after the first t-1 tokens; (ii) S is untouched; (iii) R
    runs the base recurrence with values r and rate gamma, so R_T is the final
    base state of a run with (v, beta, S0) := (r, gamma, R0)."""
    x = _inputs(seed=3)
    c = 0.5
    o, ST, RT, r = _fwd(variant, x, c, mods, return_residual=True)
    _, ST0, _ = _fwd(variant, x, c, 0)
    np.testing.assert_array_equal(ST, ST0)
    for t in range(x["q"].shape[1]):
        _, Sp, _ = _fwd(variant, _prefix(x, t), c, 0)
        p = np.einsum("hij,hi->hj", Sp[0], x["k"][0, t])
        if mods & DECAYED:
            p = np.exp(x["g"][0, t])[:, None] * p
        xr = x["v"][0, t] - p
        exp = c * np.tanh(xr / c) if mods & TANH else np.clip(xr, -c, c)
        np.testing.assert_allclose(r[0, t], exp, rtol=0, atol=1e-13)
    y = dict(x)
    y["v"], y["beta"], y["S0"] = r, x["gamma"], x["R0"]
    _, Sr, _ = _fwd(variant, y, np.inf, 0)
    np.testing.assert_allclose(RT, Sr, rtol=0, atol=1e-13)


def test_gated_delta_net_identity():
    """Table 1 (Section 2.3): Gated DeltaNet is the stateless correction of the
    decayed residual with gamma = beta, so RDN with STATELESS | DECAYED,
    gamma = beta and no clip reads o_t = S_t q_t, the updated base state
    (from the base path on the first t tokens) against q_t."""
    x = _inputs(seed=4)
    x["gamma"] = x["beta"].copy()
    o, _, _ = _fwd(RDN, x, np.inf, STATELESS | DECAYED)
    for t in range(1, x["q"].shape[1] + 1):
        _, St, _ = _fwd(RDN, _prefix(x, t), np.inf, 0)
        exp = np.einsum("hij,hi->hj", St[0], x["q"][0, t - 1])
        np.testing.assert_allclose(o[0, t - 1], exp, rtol=0, atol=1e-12)
    o0, _, _ = _fwd(RDN, x, np.inf, STATELESS)  # the undecayed residual is not GDN
    assert np.abs(o0 - o).max() > 1e-3


@pytest.mark.parametrize("variant", [RLA, RDN])
def test_decayed_T1_closed_form(variant):
    """t = 1 in the paper's d_v x d_k orientation: r = clip(v - a S0 k)."""
    x = _inputs(T=1, H=1, seed=1)
    q, k, v = x["q"][0, 0, 0], x["k"][0, 0, 0], 3.0 * x["v"][0, 0, 0]
    a, b, gm = np.exp(x["g"][0, 0, 0]), x["beta"][0, 0, 0], x["gamma"][0, 0, 0]
    S0, R0 = x["S0"][0, 0].T, x["R0"][0, 0].T  # [d_v, d_k]
    c = 0.6
    r = np.clip(v - a * S0 @ k, -c, c)
    if variant == RDN:
        R1 = a * R0 @ (np.eye(len(k)) - gm * np.outer(k, k)) + gm * np.outer(r, k)
    else:
        R1 = a * R0 + gm * np.outer(r, k)
    xx = dict(x)
    xx["v"] = v[None, None, None]
    o, _, RT = _fwd(variant, xx, c, DECAYED)
    np.testing.assert_allclose(RT[0, 0].T, R1, rtol=0, atol=1e-14)
    np.testing.assert_allclose(o[0, 0, 0], a * S0 @ q + gm * R1 @ q, rtol=0, atol=1e-14)


# ------------------------------------------------------------ PLAIN
@pytest.mark.parametrize("variant", [RLA, RDN])
def test_plain_combine_from_prefix_states(variant):
    """The plain combine changes only the read-out: the states are those of
    the method, and o_t = S_{t-1} q_t + R_t q_t with S_{t-1} the final state
    of the first t-1 tokens and R_t that of the first t."""
    x = _inputs(seed=5)
    c = 0.8
    o, ST, RT = _fwd(variant, x, c, PLAIN)
    _, ST0, RT0 = _fwd(variant, x, c, 0)
    np.testing.assert_array_equal(ST, ST0)
    np.testing.assert_array_equal(RT, RT0)
    for t in range(1, x["q"].shape[1] + 1):
        _, Sp, _ = _fwd(variant, _prefix(x, t - 1), c, 0)
        _, _, Rt = _fwd(variant, _prefix(x, t), c, 0)
        qt = x["q"][0, t - 1]
        exp = np.einsum("hij,hi->hj", Sp[0], qt) + np.einsum("hij,hi->hj", Rt[0], qt)
        np.testing.assert_allclose(o[0, t - 1], exp, rtol=0, atol=1e-12)


@pytest.mark.parametrize("variant", [RLA, RDN])
def test_plain_equals_gated_at_unit_gates(variant):
    """With a = 1 (g = 0) and gamma = 1 the two combines are the same map."""
    x = _inputs(seed=6)
    x["g"] = np.zeros_like(x["g"])
    x["gamma"] = np.ones_like(x["gamma"])
    o1, _, _ = _fwd(variant, x, 0.9, PLAIN)
    o0, _, _ = _fwd(variant, x, 0.9, 0)
    np.testing.assert_allclose(o1, o0, rtol=0, atol=1e-13)


# ------------------------------------------------------------ TANH
@pytest.mark.parametrize("variant", [RLA, RDN])
@pytest.mark.parametrize("c", [1.0, 0.4])
def test_tanh_residual_is_logcosh_descent_direction(variant, c):
    """Appendix B: the tanh residual is the negative gradient of the log-cosh
    loss c^2 log cosh((v - f)/c) with respect to the prediction f =
    S_{t-1} k_t (taken from the base path on the prefix); checked by central
    differences of the loss, elementwise."""
    x = _inputs(seed=7)
    x["v"] = 2.0 * x["v"]
    _, _, _, r = _fwd(variant, x, c, TANH, return_residual=True)
    loss = lambda f, v: c * c * np.log(np.cosh((v - f) / c))
    h = 1e-6
    for t in range(x["q"].shape[1]):
        _, Sp, _ = _fwd(variant, _prefix(x, t), c, 0)
        f = np.einsum("hij,hi->hj", Sp[0], x["k"][0, t])
        v = x["v"][0, t]
        neg_grad = -(loss(f + h, v) - loss(f - h, v)) / (2 * h)
        np.testing.assert_allclose(r[0, t], neg_grad, rtol=0, atol=1e-8)


@pytest.mark.parametrize("variant", [RLA, RDN])
def test_tanh_limits_match_clip(variant):
    """c = inf: both residuals are the identity; c = 0: both are zero."""
    x = _inputs(seed=8)
    for c in (np.inf, 0.0):
        a = _fwd(variant, x, c, TANH)
        b = _fwd(variant, x, c, 0)
        for u, w in zip(a, b):
            np.testing.assert_allclose(u, w, rtol=0, atol=1e-14)


# ------------------------------------------------------------ STATELESS
@pytest.mark.parametrize("variant", [RLA, RDN])
def test_stateless_aux_is_current_residual_outer_product(variant):
    """R_T = r_T k_T^T (rank one, from the last token alone) and nothing
    depends on R0."""
    x = _inputs(seed=9)
    c = 0.7
    o, ST, RT, r = _fwd(variant, x, c, STATELESS, return_residual=True)
    exp = np.einsum("hi,hj->hij", x["k"][0, -1], r[0, -1])
    np.testing.assert_allclose(RT[0], exp, rtol=0, atol=1e-15)
    y = dict(x)
    y["R0"] = 5.0 * x["R0"] + 1.0
    o2, ST2, RT2 = _fwd(variant, y, c, STATELESS)
    np.testing.assert_array_equal(o, o2)
    np.testing.assert_array_equal(RT, RT2)


@pytest.mark.parametrize("variant", [RLA, RDN])
def test_stateless_equals_method_without_aux_memory(variant):
    """The method with a -> 0 (g = -60) and gamma = 1 forgets R_{t-1} and
    writes R_t = r_t k_t^T: the stateless correction, exactly up to e^-60."""
    x = _inputs(seed=10)
    x["g"] = np.full_like(x["g"], -60.0)
    x["gamma"] = np.ones_like(x["gamma"])
    a = _fwd(variant, x, 0.9, STATELESS)
    b = _fwd(variant, x, 0.9, 0)
    for u, w in zip(a, b):
        np.testing.assert_allclose(u, w, rtol=0, atol=1e-12)


# ------------------------------------------------------------ gradients
MODS = [DECAYED, PLAIN, TANH, STATELESS, DECAYED | TANH, PLAIN | STATELESS]


@pytest.mark.parametrize("variant", [RLA, RDN])
@pytest.mark.parametrize("mods", MODS)
def test_variant_backward_finite_differences(variant, mods):
    """Central differences of the oracle's forward with each variant, on a few
    coordinates of every input (clip decisions kept away from c)."""
    x = _inputs(T=9, H=1, D=4, Dv=3, seed=11)
    c = 0.9
    x["v"], _ = oracle.clip_margin_condition(variant, x["q"], x["k"], x["v"], x["g"], x["beta"],
                                             x["gamma"], c, x["S0"], x["R0"], margin=1e-3,
                                             quant="f64", mods=mods)
    d = oracle.bwd(variant, x["q"], x["k"], x["v"], x["g"], x["beta"], x["gamma"], c, x["S0"],
                   x["R0"], x["dO"], dRT=np.full((1, 1, 4, 3), 0.3), mods=mods)

    def loss(y):
        o, _, RT = _fwd(variant, y, c, mods)
        return float((o * x["dO"]).sum() + 0.3 * RT.sum())

    rng = np.random.default_rng(mods)
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
