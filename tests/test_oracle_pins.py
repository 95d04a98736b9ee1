"""Pins for the fp64 oracle: checks against things the paper and the mathematics
fix, never against the oracle itself.

  * hand-worked examples (tests/golden/*.txt)
  * exact dense Kalman filter (Prop. 1) in the cases where the diagonal /
    isotropic projections are exact (axis-aligned keys, d_k = 1, one step)
  * Prop. 2 / Prop. 4 one-step projections against a numerically inverted
    dense posterior
  * the delta-rule reduction of eq. fixed-gain-approx (DeltaNet, Gated
    DeltaNet, KDA) against an independently written textbook delta rule
  * the Moebius associative scan (eq. diag-cov-scan) over random association
    trees, its fixed point, positivity and ordering invariants
  * the residual identity of eq. appendix-effective-write-residual
  * mu current-step invariance (eq. appendix-protection-current-invariance)
  * the backward pass against central finite differences and against torch
    autograd of a separately written token loop
"""
import os

import numpy as np
import pytest

import oracle
from kdn_inputs import make_inputs

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _rows(name):
    rows = []
    with open(os.path.join(GOLDEN, name)) as f:
        for line in f:
            line = line.strip()
            if line and not line.startswith("#"):
                rows.append(line.split())
    return rows


# --------------------------------------------------------------------------
# textbook algorithms written independently of the oracle


def dense_kalman(D, Om, k, v, r, S0, P0):
    """Kalman filter of Prop. 1 with dense covariance; returns per-step S, P, kappa, Shat."""
    S, P = S0.copy(), P0.copy()
    dk = P.shape[0]
    Ss, Ps, kaps, Shats = [], [], [], []
    for t in range(k.shape[0]):
        Shat = D[t] @ S
        Phat = D[t] @ P @ D[t].T + Om[t]
        gam = r[t] + k[t] @ Phat @ k[t]
        kap = Phat @ k[t] / gam
        S = Shat + np.outer(kap, v[t] - Shat.T @ k[t])
        P = (np.eye(dk) - np.outer(kap, k[t])) @ Phat
        Ss.append(S.copy()); Ps.append(P.copy()); kaps.append(kap); Shats.append(Shat)
    return np.array(Ss), np.array(Ps), np.array(kaps), np.array(Shats)


def textbook_delta_rule(alpha, beta, k, v, q, S0, tau):
    """S_t = (I - beta k k^T) diag(alpha) S_{t-1} + beta k v^T, o = tau S^T q (eq. unified-delta-rule)."""
    S = S0.copy()
    dk = S.shape[0]
    os_ = []
    for t in range(k.shape[0]):
        S = (np.eye(dk) - beta[t] * np.outer(k[t], k[t])) @ (np.diag(alpha[t]) @ S) \
            + beta[t] * np.outer(k[t], v[t])
        os_.append(tau * S.T @ q[t])
    return np.array(os_), S


def run_steps(variant, ins, mu=None, scale=None):
    """Token-by-token decode calls; returns per-token S_t and p_t (states after t)."""
    S = ins.get("S0")
    p = ins.get("p0")
    B, T, H, dk = ins["q"].shape
    dv = ins["v"].shape[-1]
    if S is None:
        S = np.zeros((B, H, dk, dv))
    if p is None:
        p = np.ones((B, H, dk) if variant == "diag" else (B, H))
    Ss, ps, os_ = [], [], []
    for t in range(T):
        sl = {n: ins[n][:, t] for n in ("q", "k", "v", "g", "omega", "r")}
        o, S, p = oracle.decode_step(variant, sl["q"], sl["k"], sl["v"], sl["g"], sl["omega"],
                                     sl["r"], S, p, mu=mu, scale=scale)
        Ss.append(S); ps.append(p); os_.append(o)
    return np.array(Ss), np.array(ps), np.array(os_)


# --------------------------------------------------------------------------
# golden worked examples


@pytest.mark.parametrize("variant", ["diag", "iso"])
def test_golden_scalar_kalman(variant):
    rows = _rows("scalar_kf_worked.txt")
    for case in ("A", "B"):
        rs = [r for r in rows if r[0] == case]
        T = len(rs)
        col = lambda i: np.array([float(r[i]) for r in rs])
        g, om, rr, v = col(2), col(3), col(4), col(5)
        kap_ref, o_ref, S_ref, p_ref = col(6), col(7), col(8), col(9)
        S0 = np.zeros((1, 1, 1, 1)) if case == "A" else np.ones((1, 1, 1, 1))
        p0 = np.ones((1, 1, 1)) if variant == "diag" else np.ones((1, 1))
        ones = np.ones((1, T, 1, 1))
        gg = g.reshape(1, T, 1, 1)
        w = om.reshape(1, T, 1, 1) if variant == "diag" else om.reshape(1, T, 1)
        res = oracle.fwd(variant, ones, ones, v.reshape(1, T, 1, 1), gg, w, rr.reshape(1, T, 1),
                         S0, p0, mu=1.0, scale=1.0, trace=True)
        np.testing.assert_allclose(res["o"].ravel(), o_ref, rtol=1e-14, atol=1e-15)
        np.testing.assert_allclose(res["kappa"].ravel(), kap_ref, rtol=1e-14)
        np.testing.assert_allclose(res["ST"].ravel(), S_ref[-1:], rtol=1e-14)
        np.testing.assert_allclose(np.ravel(res["p"]), p_ref, rtol=1e-14)


def test_golden_iso_worked():
    rows = _rows("iso_worked.txt")
    T = len(rows)
    a = np.array([[float(x) for x in r] for r in rows])
    k = a[:, 1:3].reshape(1, T, 1, 2)
    v = a[:, 3].reshape(1, T, 1, 1)
    q = np.ones((1, T, 1, 2))
    g = np.zeros((1, T, 1))
    om = np.ones((1, T, 1))
    rr = np.ones((1, T, 1))
    res = oracle.fwd("iso", q, k, v, g, om, rr, None, None, mu=1.0, scale=1.0, trace=True)
    np.testing.assert_allclose(res["o"].ravel(), a[:, 5], rtol=1e-12)
    beta = res["kappa"][0, :, 0, :] / a[:, 1:3].clip(min=1e-300)
    np.testing.assert_allclose(np.where(a[:, 1:3] > 0, beta, a[:, 4:5]), np.repeat(a[:, 4:5], 2, 1),
                               rtol=1e-12)
    np.testing.assert_allclose(res["ST"].ravel(), a[-1, 6:8], rtol=1e-12)
    np.testing.assert_allclose(np.ravel(res["p"]), a[:, 8], rtol=1e-12)


def test_golden_balanced_key():
    """P7: one mu-scaled update from phat_i = p on a balanced key of support m."""
    for r_ in _rows("balanced_key.txt"):
        m, r, p, mu, Vp, Ve = int(r_[0]), *map(float, r_[1:])
        dk = m + 3  # extra channels carry no key energy
        k = np.zeros((1, 1, 1, dk))
        k[..., :m] = 1.0 / np.sqrt(m)
        q = np.zeros_like(k)
        v = np.ones((1, 1, 1, 2))
        g = np.zeros((1, 1, 1, dk))
        om = np.full((1, 1, 1, dk), p / 2)
        p0 = np.full((1, 1, dk), p / 2)            # phat = 1 * p/2 + p/2 = p
        res = oracle.fwd("diag", q, k, v, g, om, np.full((1, 1, 1), r), None, p0, mu=mu)
        kk = k.ravel()
        V_proj = float(np.sum(kk * kk * res["pT"].ravel()))
        assert V_proj == pytest.approx(Vp, rel=1e-13)
        # exact posterior along k: k^T P* k with P* = (I - kappa k^T) diag(phat)
        Phat = np.diag(np.full(dk, p))
        kap = Phat @ kk / (r + kk @ Phat @ kk)
        Pstar = (np.eye(dk) - np.outer(kap, kk)) @ Phat
        assert float(kk @ Pstar @ kk) == pytest.approx(Ve, rel=1e-13)


# --------------------------------------------------------------------------
# P1: exact Kalman filter where the projection is exact


def _rand_diag_problem(rng, T, dk, dv, axis_aligned):
    k = np.zeros((T, dk))
    if axis_aligned:
        idx = rng.integers(0, dk, size=T)
        k[np.arange(T), idx] = rng.uniform(0.3, 2.0, size=T) * rng.choice([-1, 1], size=T)
    else:
        k = rng.standard_normal((T, dk))
    return dict(k=k, q=rng.standard_normal((T, dk)), v=rng.standard_normal((T, dv)),
                g=np.log(rng.uniform(0.5, 0.99, size=(T, dk))),
                om=rng.uniform(0.05, 0.5, size=(T, dk)), r=rng.uniform(0.2, 2.0, size=T),
                S0=rng.standard_normal((dk, dv)) * 0.3, p0=rng.uniform(0.5, 2.0, size=dk))


def test_p1_axis_aligned_keys_equal_exact_kf():
    rng = np.random.default_rng(1)
    T, dk, dv = 40, 6, 3
    P = _rand_diag_problem(rng, T, dk, dv, axis_aligned=True)
    al = np.exp(P["g"])
    Ss, Ps, _, _ = dense_kalman(np.array([np.diag(a) for a in al]),
                                np.array([np.diag(w) for w in P["om"]]),
                                P["k"], P["v"], P["r"], P["S0"], np.diag(P["p0"]))
    ins = dict(q=P["q"][None, :, None], k=P["k"][None, :, None], v=P["v"][None, :, None],
               g=P["g"][None, :, None], omega=P["om"][None, :, None], r=P["r"][None, :, None],
               S0=P["S0"][None, None], p0=P["p0"][None, None])
    S_o, p_o, o_o = run_steps("diag", ins, mu=1.0, scale=0.7)
    np.testing.assert_allclose(S_o[:, 0, 0], Ss, rtol=1e-11, atol=1e-12)
    np.testing.assert_allclose(p_o[:, 0, 0], np.array([np.diag(x) for x in Ps]), rtol=1e-11)
    # off-diagonals of the exact posterior stay zero in this case
    assert np.max(np.abs(Ps - np.array([np.diag(np.diag(x)) for x in Ps]))) < 1e-14
    np.testing.assert_allclose(o_o[:, 0, 0], 0.7 * np.einsum("tij,ti->tj", Ss, P["q"]),
                               rtol=1e-11, atol=1e-12)


def test_p1_scalar_key_dim_all_equal_exact_kf():
    rng = np.random.default_rng(2)
    T, dv = 30, 4
    P = _rand_diag_problem(rng, T, 1, dv, axis_aligned=False)
    al = np.exp(P["g"])
    Ss, Ps, _, _ = dense_kalman(al[:, :, None], P["om"][:, :, None], P["k"], P["v"], P["r"],
                                P["S0"], np.diag(P["p0"]))
    base = dict(q=P["q"][None, :, None], k=P["k"][None, :, None], v=P["v"][None, :, None],
                r=P["r"][None, :, None], S0=P["S0"][None, None])
    d = oracle.fwd("diag", base["q"], base["k"], base["v"], P["g"][None, :, None],
                   P["om"][None, :, None], base["r"], base["S0"], P["p0"][None, None], mu=1.0,
                   trace=True)
    i = oracle.fwd("iso", base["q"], base["k"], base["v"], P["g"][None, :, None, 0],
                   P["om"][None, :, None, 0], base["r"], base["S0"], P["p0"][None, None], mu=1.0,
                   trace=True)
    np.testing.assert_allclose(d["ST"][0, 0], Ss[-1], rtol=1e-11, atol=1e-13)
    np.testing.assert_allclose(i["ST"][0, 0], Ss[-1], rtol=1e-11, atol=1e-13)
    np.testing.assert_allclose(d["p"][0, :, 0, 0], Ps[:, 0, 0], rtol=1e-11)
    np.testing.assert_allclose(i["p"][0, :, 0], Ps[:, 0, 0], rtol=1e-11)
    np.testing.assert_allclose(d["o"], i["o"], rtol=1e-12, atol=1e-14)


# --------------------------------------------------------------------------
# P2 / P3: one-step variational projections


def test_p2_prop2_one_step_diag():
    rng = np.random.default_rng(3)
    dk, dv = 7, 3
    for _ in range(5):
        P = _rand_diag_problem(rng, 1, dk, dv, axis_aligned=False)
        al = np.exp(P["g"][0])
        Ss, Ps, _, _ = dense_kalman(np.diag(al)[None], np.diag(P["om"][0])[None], P["k"],
                                    P["v"], P["r"], P["S0"], np.diag(P["p0"]))
        res = oracle.fwd("diag", P["q"][None, :, None], P["k"][None, :, None],
                         P["v"][None, :, None], P["g"][None, :, None], P["om"][None, :, None],
                         P["r"][None, :, None], P["S0"][None, None], P["p0"][None, None], mu=1.0)
        np.testing.assert_allclose(res["ST"][0, 0], Ss[0], rtol=1e-11, atol=1e-13)
        p_var = 1.0 / np.diag(np.linalg.inv(Ps[0]))       # reverse-KL diagonal projection
        np.testing.assert_allclose(res["pT"][0, 0], p_var, rtol=1e-11)


def test_p3_prop4_one_step_iso():
    rng = np.random.default_rng(4)
    dk, dv = 6, 2
    for _ in range(5):
        k = rng.standard_normal((1, dk))
        v = rng.standard_normal((1, dv))
        q = rng.standard_normal((1, dk))
        a = rng.uniform(0.5, 0.99)
        om, r, b0 = rng.uniform(0.05, 0.5), rng.uniform(0.2, 2.0), rng.uniform(0.5, 2.0)
        S0 = rng.standard_normal((dk, dv)) * 0.3
        Ss, Ps, _, _ = dense_kalman((a * np.eye(dk))[None], (om * np.eye(dk))[None], k, v,
                                    np.array([r]), S0, b0 * np.eye(dk))
        res = oracle.fwd("iso", q[None, :, None], k[None, :, None], v[None, :, None],
                         np.full((1, 1, 1), np.log(a)), np.full((1, 1, 1), om),
                         np.full((1, 1, 1), r), S0[None, None], np.full((1, 1), b0), mu=1.0)
        np.testing.assert_allclose(res["ST"][0, 0], Ss[0], rtol=1e-11, atol=1e-13)
        b_harm = dk / np.trace(np.linalg.inv(Ps[0]))      # harmonic mean of eigenvalues
        assert res["pT"][0, 0] == pytest.approx(b_harm, rel=1e-12)


# --------------------------------------------------------------------------
# P4: delta-rule reduction in surrogate mode


@pytest.mark.parametrize("kind", ["deltanet", "gated_deltanet", "kda"])
def test_p4_surrogate_reduces_to_delta_rule(kind):
    rng = np.random.default_rng(5)
    T, dk, dv = 25, 5, 3
    k = rng.standard_normal((T, dk))
    k /= np.linalg.norm(k, axis=1, keepdims=True) * rng.uniform(0.7, 1.3, size=(T, 1))
    q = rng.standard_normal((T, dk))
    v = rng.standard_normal((T, dv))
    r = rng.uniform(0.2, 2.0, size=T)
    n2 = np.sum(k * k, axis=1)
    beta = rng.uniform(0.05, 0.95, size=T) / n2
    if kind == "deltanet":
        alpha = np.ones((T, dk))
    elif kind == "gated_deltanet":
        alpha = np.repeat(rng.uniform(0.6, 0.99, size=(T, 1)), dk, axis=1)
    else:
        alpha = rng.uniform(0.6, 0.99, size=(T, dk))
    S0 = rng.standard_normal((dk, dv)) * 0.5
    o_ref, S_ref = textbook_delta_rule(alpha, beta, k, v, q, S0, 0.5)
    bhat = beta * r / (1.0 - beta * n2)  # predicted variance that yields this beta
    res = oracle.fwd("iso", q[None, :, None], k[None, :, None], v[None, :, None],
                     np.log(alpha)[None, :, None], np.ones((1, T, 1)), r[None, :, None],
                     S0[None, None], None, bhat=bhat[None, :, None], scale=0.5)
    np.testing.assert_allclose(res["o"][0, :, 0], o_ref, rtol=1e-11, atol=1e-12)
    np.testing.assert_allclose(res["ST"][0, 0], S_ref, rtol=1e-11, atol=1e-12)


# --------------------------------------------------------------------------
# P5: Moebius associative scan, invariants, fixed point


def _mobius_mats(alpha2, omega, u):
    M = np.empty(alpha2.shape + (2, 2))
    M[..., 0, 0] = alpha2
    M[..., 0, 1] = omega
    M[..., 1, 0] = u * alpha2
    M[..., 1, 1] = 1.0 + u * omega
    return M


def _tree_prod(M, lo, hi, rng, renorm):
    """Ordered product M[hi-1] ... M[lo] over a random association tree."""
    if hi - lo == 1:
        return M[lo].copy()
    mid = int(rng.integers(lo + 1, hi))
    P = _tree_prod(M, mid, hi, rng, renorm) @ _tree_prod(M, lo, mid, rng, renorm)
    if renorm:
        P /= np.max(np.abs(P))
    return P


@pytest.mark.parametrize("renorm", [False, True])
def test_p5_mobius_scan_matches_recursion(renorm):
    ins = make_inputs("diag", 1, 48, 2, 8, 4, dtype="f32", seed=11, p0_range=(0.5, 2.0))
    mu = 8.0
    res = oracle.fwd("diag", ins["q"], ins["k"], ins["v"], ins["g"], ins["omega"], ins["r"],
                     None, ins["p0"], mu=mu, trace=True)
    rng = np.random.default_rng(7)
    alpha2 = np.exp(2 * ins["g"])
    u = mu * ins["k"] ** 2 / ins["r"][..., None]
    M = _mobius_mats(alpha2, ins["omega"], u)           # [B,T,H,dk,2,2]
    for h in range(2):
        for i in range(8):
            z0 = np.array([ins["p0"][0, h, i], 1.0])
            for t in range(48):
                P = _tree_prod(M[0, :, h, i], 0, t + 1, rng, renorm)
                z = P @ z0
                assert z[0] / z[1] == pytest.approx(res["p"][0, t, h, i], rel=1e-12)
    # invariants: positivity, omega <= phat, p <= phat, 0 <= beta_eff < 1
    assert np.all(res["p"] > 0)
    assert np.all(res["phat"] >= ins["omega"] * (1 - 1e-15))
    assert np.all(res["p"] <= res["phat"] * (1 + 1e-15))
    beff = np.sum(ins["k"] * res["kappa"], axis=-1)
    assert np.all(beff >= 0) and np.all(beff < 1)


def test_p5_fixed_point_constant_inputs():
    T, dk = 600, 3
    a2, om, r, mu = np.array([0.81, 0.5, 0.95]), np.array([0.1, 0.3, 0.02]), 0.7, 2.0
    k = np.array([0.6, 0.0, 0.8])
    ones = np.ones((1, T, 1, 1))
    res = oracle.fwd("diag", ones * np.ones(dk), ones * k, ones * np.ones(2),
                     ones * (0.5 * np.log(a2)), ones * om, np.full((1, T, 1), r), None, None,
                     mu=mu)
    u = mu * k * k / r
    # positive root of u a2 p^2 + (1 + u om - a2) p - om = 0 (u = 0: p = om / (1 - a2))
    with np.errstate(divide="ignore", invalid="ignore"):
        bq = 1 + u * om - a2
        root = np.where(u > 0, (-bq + np.sqrt(bq * bq + 4 * u * a2 * om)) / (2 * u * a2),
                        om / (1 - a2))
    np.testing.assert_allclose(res["pT"][0, 0], root, rtol=1e-12)


# --------------------------------------------------------------------------
# P6 residual identity, P8 mu invariance, state hand-off


@pytest.mark.parametrize("variant", ["diag", "iso"])
def test_p6_residual_identity(variant):
    ins = make_inputs(variant, 2, 20, 2, 6, 3, dtype="f32", seed=3, s0_std=0.5)
    S_o, _, _ = run_steps(variant, ins)
    res = oracle.fwd(variant, ins["q"], ins["k"], ins["v"], ins["g"], ins["omega"], ins["r"],
                     ins["S0"], None, trace=True)
    alpha = np.exp(ins["g"])
    if alpha.ndim == 3:
        alpha = np.repeat(alpha[..., None], 6, axis=-1)
    Sprev = np.concatenate([ins["S0"][None], S_o[:-1]], axis=0)   # [T,B,H,dk,dv]
    for t in range(20):
        k = ins["k"][:, t]
        v = ins["v"][:, t]
        Shat = alpha[:, t, :, :, None] * Sprev[t]
        lhs = v - np.einsum("bhij,bhi->bhj", S_o[t], k)
        beff = np.sum(k * res["kappa"][:, t], axis=-1)
        rhs = (1 - beff)[..., None] * (v - np.einsum("bhij,bhi->bhj", Shat, k))
        np.testing.assert_allclose(lhs, rhs, rtol=1e-10, atol=1e-12)


@pytest.mark.parametrize("variant", ["diag", "iso"])
def test_p8_mu_current_step_invariance(variant):
    ins = make_inputs(variant, 1, 6, 2, 8, 4, dtype="f32", seed=9, s0_std=0.3)
    args = [ins[n] for n in ("q", "k", "v", "g", "omega", "r")]
    a = oracle.fwd(variant, *args, ins["S0"], None, mu=1.0, trace=True)
    b = oracle.fwd(variant, *args, ins["S0"], None, mu=8.0, trace=True)
    np.testing.assert_array_equal(a["o"][:, 0], b["o"][:, 0])
    np.testing.assert_array_equal(a["kappa"][:, 0], b["kappa"][:, 0])
    assert np.max(np.abs(a["o"][:, 1:] - b["o"][:, 1:])) > 1e-6
    # d p_1 / d mu = -(k^2/r) p_1^2  (diag)  or  -(|k|^2/(dk r)) b_1^2  (iso)
    h = 1e-6
    c = oracle.fwd(variant, *args, ins["S0"], None, mu=8.0 + h, trace=True)
    d = oracle.fwd(variant, *args, ins["S0"], None, mu=8.0 - h, trace=True)
    fd = (c["p"][:, 0] - d["p"][:, 0]) / (2 * h)
    k = ins["k"][:, 0]
    r = ins["r"][:, 0]
    if variant == "diag":
        an = -(k * k / r[..., None]) * b["p"][:, 0] ** 2
    else:
        an = -(np.sum(k * k, -1) / (8 * r)) * b["p"][:, 0] ** 2
    np.testing.assert_allclose(fd, an, rtol=1e-6, atol=1e-7 * np.max(np.abs(an)))


@pytest.mark.parametrize("variant", ["diag", "iso"])
def test_state_handoff_and_decode_equal_prefill(variant):
    ins = make_inputs(variant, 2, 30, 2, 5, 3, dtype="f32", seed=21, s0_std=0.1,
                      p0_range=(0.5, 2.0))
    args = [ins[n] for n in ("q", "k", "v", "g", "omega", "r")]
    full = oracle.fwd(variant, *args, ins["S0"], ins["p0"])
    a = oracle.fwd(variant, *[x[:, :13] for x in args], ins["S0"], ins["p0"])
    b = oracle.fwd(variant, *[x[:, 13:] for x in args], a["ST"], a["pT"])
    np.testing.assert_allclose(np.concatenate([a["o"], b["o"]], 1), full["o"], rtol=1e-13,
                               atol=1e-15)
    np.testing.assert_allclose(b["ST"], full["ST"], rtol=1e-13, atol=1e-15)
    S_o, p_o, o_o = run_steps(variant, ins)
    np.testing.assert_allclose(np.moveaxis(o_o, 0, 1), full["o"], rtol=1e-13, atol=1e-15)
    np.testing.assert_allclose(p_o[-1], full["pT"], rtol=1e-13)


# --------------------------------------------------------------------------
# P9: backward


def _loss_fn(variant, base, wo, wS, wp, mu):
    def f(ins):
        res = oracle.fwd(variant, ins["q"], ins["k"], ins["v"], ins["g"], ins["omega"],
                         ins["r"], ins["S0"], ins["p0"], mu=mu)
        return (np.sum(wo * res["o"]) + np.sum(wS * res["ST"]) + np.sum(wp * res["pT"]))
    return f


@pytest.mark.parametrize("variant,per_channel", [("diag", True), ("iso", True), ("iso", False)])
def test_p9_backward_finite_differences(variant, per_channel):
    B, T, H, dk, dv = 1, 9, 2, 3, 2
    ins = make_inputs(variant, B, T, H, dk, dv, dtype="f32", seed=31, s0_std=0.4,
                      p0_range=(0.5, 2.0), per_channel_decay=per_channel, with_grad=True)
    rng = np.random.default_rng(8)
    wS = rng.standard_normal((B, H, dk, dv))
    wp = rng.standard_normal(ins["p0"].shape)
    mu = 2.5
    f = _loss_fn(variant, ins, ins["dO"], wS, wp, mu)
    an = oracle.bwd(variant, ins["q"], ins["k"], ins["v"], ins["g"], ins["omega"], ins["r"],
                    ins["S0"], ins["p0"], ins["dO"], wS, wp, mu=mu)
    names = {"q": "dq", "k": "dk", "v": "dv", "g": "dg", "omega": "domega", "r": "dr",
             "S0": "dS0", "p0": "dp0"}
    h = 1e-6
    for n, gn in names.items():
        x = ins[n]
        fd = np.zeros_like(x)
        for idx in np.ndindex(x.shape):
            xp = dict(ins); xp[n] = x.copy(); xp[n][idx] += h
            xm = dict(ins); xm[n] = x.copy(); xm[n][idx] -= h
            fd[idx] = (f(xp) - f(xm)) / (2 * h)
        err = np.max(np.abs(fd - an[gn])) / max(np.max(np.abs(fd)), 1e-30)
        assert err < 1e-6, (n, err)
    # the information scale mu (one value shared by all sequences): sum of dmu
    fd_mu = (_loss_fn(variant, ins, ins["dO"], wS, wp, mu + h)(ins)
             - _loss_fn(variant, ins, ins["dO"], wS, wp, mu - h)(ins)) / (2 * h)
    assert abs(fd_mu - an["dmu"].sum()) <= 1e-6 * abs(fd_mu), (fd_mu, an["dmu"].sum())


@pytest.mark.parametrize("variant,per_channel", [("diag", True), ("iso", True), ("iso", False)])
def test_p9_backward_matches_torch_autograd(variant, per_channel):
    torch = pytest.importorskip("torch")
    B, T, H, dk, dv = 2, 70, 1, 4, 3  # crosses the oracle's 64-token checkpoint
    ins = make_inputs(variant, B, T, H, dk, dv, dtype="f32", seed=41, s0_std=0.4,
                      p0_range=(0.5, 2.0), per_channel_decay=per_channel, with_grad=True)
    mu, tau = 4.0, 0.5
    tt = {n: torch.tensor(ins[n], dtype=torch.float64, requires_grad=True)
          for n in ("q", "k", "v", "g", "omega", "r", "S0", "p0")}
    # token loop written with torch ops, independently of the C oracle
    outs = []
    S, p = tt["S0"], tt["p0"]
    for t in range(T):
        k, q, v, r = tt["k"][:, t], tt["q"][:, t], tt["v"][:, t], tt["r"][:, t]
        al = torch.exp(tt["g"][:, t])
        if not per_channel:
            al = al[..., None].expand(B, H, dk)
        if variant == "diag":
            ph = al ** 2 * p + tt["omega"][:, t]
            kap = ph * k / (r + (ph * k * k).sum(-1))[..., None]
        else:
            ph = (al ** 2).mean(-1) * p + tt["omega"][:, t]
            kap = (ph / (r + ph * (k * k).sum(-1)))[..., None] * k
        Sh = al[..., None] * S
        delta = v - torch.einsum("bhij,bhi->bhj", Sh, k)
        S = Sh + kap[..., None] * delta[..., None, :]
        outs.append(tau * torch.einsum("bhij,bhi->bhj", S, q))
        if variant == "diag":
            u = mu * k * k / r[..., None]
        else:
            u = mu * (k * k).sum(-1) / (dk * r)
        p = ph / (1 + u * ph)
    o = torch.stack(outs, 1)
    rng = np.random.default_rng(2)
    wS = rng.standard_normal(S.shape)
    wp = rng.standard_normal(p.shape)
    L = (o * torch.tensor(ins["dO"])).sum() + (S * torch.tensor(wS)).sum() + \
        (p * torch.tensor(wp)).sum()
    L.backward()
    an = oracle.bwd(variant, ins["q"], ins["k"], ins["v"], ins["g"], ins["omega"], ins["r"],
                    ins["S0"], ins["p0"], ins["dO"], wS, wp, mu=mu, scale=tau)
    for n, gn in (("q", "dq"), ("k", "dk"), ("v", "dv"), ("g", "dg"), ("omega", "domega"),
                  ("r", "dr"), ("S0", "dS0"), ("p0", "dp0")):
        np.testing.assert_allclose(an[gn], tt[n].grad.numpy(), rtol=1e-9, atol=1e-12,
                                   err_msg=n)


# --------------------------------------------------------------------------
# Gate parameterisation (eq. kla-box-parameterization): logits in, logit gradients out


def _logit_inputs(variant, per_channel, seed):
    """Logits whose activations look like the workload's gates: x ~ N(2, 1) for the
    decay, y, z ~ N(0, 1) for the noises."""
    ins = make_inputs(variant, 1, 9, 2, 3, 2, dtype="f32", seed=seed, s0_std=0.4,
                      p0_range=(0.5, 2.0), per_channel_decay=per_channel, with_grad=True)
    rng = np.random.default_rng(seed + 1)
    ins["g"] = rng.normal(2.0, 1.0, ins["g"].shape)
    ins["omega"] = rng.normal(0.0, 1.0, ins["omega"].shape)
    ins["r"] = rng.normal(0.0, 1.0, ins["r"].shape)
    return ins


def test_gate_activations_special_values():
    """sigmoid(0) = 1/2, softplus(0) = log 2, softplus(z) -> z for large z and
    -> e^z for very negative z, r_min the floor of r; log alpha <= 0."""
    x = np.array([0.0, 40.0, -40.0, 3.0])
    g, w, r = oracle.gates_from_logits(x, x, x, 0.01)
    assert np.allclose(np.exp(g), [0.5, 1.0, np.exp(-40.0), 1 / (1 + np.exp(-3.0))], rtol=1e-14,
                       atol=0)
    assert np.allclose(w, [np.log(2.0), 40.0, np.exp(-40.0), np.log1p(np.exp(3.0))], rtol=1e-14)
    assert np.allclose(r - 0.01, w, rtol=1e-14) and np.all(r > 0.01) and np.all(g <= 0)


@pytest.mark.parametrize("variant,per_channel", [("diag", True), ("iso", True), ("iso", False)])
def test_gate_logits_backward_finite_differences(variant, per_channel):
    """The logit gradients (the adjoint through sigmoid / softplus / r_min +
    softplus) agree with central differences of the logit-mode forward."""
    ins = _logit_inputs(variant, per_channel, 53)
    rng = np.random.default_rng(9)
    wS = rng.standard_normal(ins["S0"].shape)
    wp = rng.standard_normal(ins["p0"].shape)

    def f(d):
        res = oracle.fwd(variant, d["q"], d["k"], d["v"], d["g"], d["omega"], d["r"], d["S0"],
                         d["p0"], gates="logits", r_min=0.05)
        return np.sum(ins["dO"] * res["o"]) + np.sum(wS * res["ST"]) + np.sum(wp * res["pT"])

    an = oracle.bwd(variant, ins["q"], ins["k"], ins["v"], ins["g"], ins["omega"], ins["r"],
                    ins["S0"], ins["p0"], ins["dO"], wS, wp, gates="logits", r_min=0.05)
    h = 1e-6
    for n, gn in (("g", "dg"), ("omega", "domega"), ("r", "dr"), ("k", "dk")):
        x = ins[n]
        fd = np.zeros_like(x)
        for idx in np.ndindex(x.shape):
            xp = dict(ins); xp[n] = x.copy(); xp[n][idx] += h
            xm = dict(ins); xm[n] = x.copy(); xm[n][idx] -= h
            fd[idx] = (f(xp) - f(xm)) / (2 * h)
        err = np.max(np.abs(fd - an[gn])) / max(np.max(np.abs(fd)), 1e-30)
        assert err < 1e-6, (n, err)
