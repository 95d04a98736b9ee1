"""App. F's chunkwise algorithm in fp64, against the oracle's token loop.

The fused kernels compute the chunked form of App. F, not the token loop, and
the Diagonal forward computes it in a rearranged order.  These CPU tests check,
in float64 with numpy, that both are exact rewrites of the recurrence the
oracle steps through token by token (Prop. 3 / Prop. 5), so that the GPU
parity tests only measure rounding:

  * the chunked form as App. F states it: gain chunks of C_g tokens (the
    Moebius summary of each chunk and channel, eq. chunk-gain-summary; the
    exclusive carry, eq. chunk-gain-carry; the replay and the gain emitted from
    the pre-write state, eqs. chunk-gain-local-prefix and chunk-gain-emission)
    and, independently, memory chunks of C_m tokens (eqs.
    chunk-memory-normalization to chunk-memory-output-state);
  * the order the Diagonal forward uses: intra-chunk decay ratios referenced at
    the middle of the chunk's log-decay range, with a direct form past
    G_C < -160; the solve as A = diag(s) L^-1 with L = diag(s) +
    strict_lower(T'); R = A (V - Kbar S_in); outputs and state from
    R' = diag(1/s) R and the unnormalised A'_qk and K'.

The same is done for the backward (the chunk adjoint of the fused backward,
its stages B1-B10 and the scalings by Gamma, then the gain adjoint token by
token, against the oracle's gradients) and for the join of the
sequence-parallel forward (a two-level scan of Moebius summaries for the
uncertainty entering each segment; per segment the memory from 0 and the
transition Phi; S_in(j+1) = Phi_j S_in(j) + Sv_j).

Nothing here runs on, or is shared with, the CUDA path.
"""
import numpy as np
import pytest

import oracle
from kdn_inputs import make_inputs

TOL = 1e-9  # max |chunked - token loop| / RMS(token loop), float64 throughout


@pytest.fixture(scope="module", autouse=True)
def _built():
    oracle.build()


def _rel(x, ref):
    return float(np.max(np.abs(x - ref)) / np.sqrt(np.mean(ref * ref)))


def _renorm(z):
    # n/d is unchanged by a common factor: divide by the largest magnitude
    m = np.max(np.abs(z.reshape(z.shape[0], -1)), axis=1)
    return z / m.reshape((-1,) + (1,) * (z.ndim - 1))


# ---------------------------------------------------------------------------
# App. F.1: chunkwise gain

def gain_chunked(variant, k, g, omega, r, p0, mu, Cg):
    """kappa [T, dk], phat [T, P] and p_T [P] of one sequence, by gain chunks of
    Cg tokens (P = dk channels for the Diagonal KDN, 1 for the Isotropic)."""
    T, dk = k.shape
    if variant == "diag":
        a = np.exp(2.0 * g)                                  # alpha^2 per channel
        u = mu * k * k / r[:, None]                          # eq. diag-cov-update
        w = omega
    else:
        a = (np.mean(np.exp(2.0 * g), axis=1) if g.ndim == 2 else np.exp(2.0 * g))[:, None]
        u = (mu * np.sum(k * k, axis=1) / (dk * r))[:, None]  # Prop. 5
        w = omega[:, None]
    P = a.shape[1]
    # token matrices M_t = [[a, w], [u a, 1 + u w]] (eq. diag-cov-scan), [T, P, 2, 2]
    M = np.empty((T, P, 2, 2))
    M[:, :, 0, 0], M[:, :, 0, 1] = a, w
    M[:, :, 1, 0], M[:, :, 1, 1] = u * a, 1.0 + u * w
    starts = list(range(0, T, Cg))
    # summaries, later tokens on the left (eq. chunk-gain-summary)
    summ = []
    for c0 in starts:
        prod = np.broadcast_to(np.eye(2), (P, 2, 2)).copy()
        for t in range(c0, min(c0 + Cg, T)):
            prod = _renorm(np.einsum("pij,pjk->pik", M[t], prod))
        summ.append(prod)
    # exclusive carry from z_0 = [p_0, 1] (eq. chunk-gain-carry)
    z = np.stack([np.broadcast_to(p0, (P,)), np.ones(P)], axis=1)
    carry = []
    for prod in summ:
        carry.append(z)
        z = _renorm(np.einsum("pij,pj->pi", prod, z))
    p_T = z[:, 0] / z[:, 1]
    # replay every chunk from its carry; the gain reads the pre-write state
    phat = np.empty((T, P))
    for c0, zin in zip(starts, carry):
        z = zin
        for t in range(c0, min(c0 + Cg, T)):
            phat[t] = a[t] * (z[:, 0] / z[:, 1]) + w[t]      # eq. chunk-gain-emission
            z = _renorm(np.einsum("pij,pj->pi", M[t], z))
    if variant == "diag":
        s = r + np.sum(phat * k * k, axis=1)
        kappa = phat * k / s[:, None]
    else:
        beta = phat[:, 0] / (r + phat[:, 0] * np.sum(k * k, axis=1))
        kappa = beta[:, None] * k
    return kappa, phat, p_T


# ---------------------------------------------------------------------------
# App. F.2: chunkwise memory, as printed

def memory_chunked(q, k, v, G, kappa, S0, tau, Cm):
    """o [T, dv] and S_T of one sequence, by memory chunks of Cm tokens; G [T, dk]
    is log alpha per channel."""
    T, dk = k.shape
    S = S0.copy()
    o = np.empty((T, v.shape[1]))
    for c0 in range(0, T, Cm):
        sl = slice(c0, min(c0 + Cm, T))
        C = sl.stop - sl.start
        gam = np.exp(np.cumsum(G[sl], axis=0))               # gamma_r, r = 1..C
        K, Kk, Q, V = k[sl], kappa[sl], q[sl], v[sl]
        Kbar, Kkbar, Qbar = gam * K, Kk / gam, tau * gam * Q  # eq. chunk-memory-scaled-keys
        Tm = np.tril(Kbar @ Kkbar.T, -1)
        A = np.linalg.inv(np.eye(C) + Tm)                    # eq. chunk-memory-wy
        W, U = A @ Kbar, A @ V
        R = U - W @ S
        Ktail = (gam[-1] / gam) * Kk                          # eq. chunk-memory-tail-output
        Aqk = np.tril(Qbar @ Kkbar.T)
        o[sl] = Qbar @ S + Aqk @ R                            # eq. chunk-memory-output-state
        S = gam[-1][:, None] * S + Ktail.T @ R
    return o, S


# ---------------------------------------------------------------------------
# the order of the Diagonal forward kernel

RANGE_G = -160.0  # a chunk with G_C below this in some channel forms its ratios directly


def memory_kernel_order(q, k, v, G, phat, r, S0, tau, Cm=64):
    """o, S_T of one Diagonal-KDN sequence in the forward kernel's order.
    Returns also the number of chunks that took the direct (range) form."""
    T, dk = k.shape
    S = S0.copy()
    o = np.empty((T, v.shape[1]))
    n_range = 0
    for c0 in range(0, T, Cm):
        sl = slice(c0, min(c0 + Cm, T))
        C = sl.stop - sl.start
        Gc = np.cumsum(G[sl], axis=0)
        GC = Gc[-1]
        K, Q, V, ph = k[sl], q[sl], v[sl], phat[sl]
        if np.all(GC >= RANGE_G):
            c = GC / 2.0                                       # middle of the decay range
            Kb1, Qb1 = K * np.exp(Gc - c), tau * Q * np.exp(Gc - c)
            Kk1 = ph * K * np.exp(c - Gc)
            # the referenced factors stay inside float32's range
            assert np.max(np.abs(Gc - c)) <= 80.0 + 1e-9
            Tp, Ap = Kb1 @ Kk1.T, Qb1 @ Kk1.T
        else:
            n_range += 1
            ratio = np.exp(np.minimum(Gc[:, None, :] - Gc[None, :, :], 0.0))  # [t, s, i], <= 1
            Tp = np.einsum("ti,si,tsi->ts", K, ph * K, ratio)
            Ap = tau * np.einsum("ti,si,tsi->ts", Q, ph * K, ratio)
        s = r[sl] + np.diag(Tp)                               # eq. kla-box-gain, from T'
        L = np.diag(s) + np.tril(Tp, -1)
        A = np.diag(s) @ np.linalg.inv(L)                     # = (I + T)^-1
        gam = np.exp(Gc)
        R = A @ (V - (gam * K) @ S)
        Rp = R / s[:, None]
        Kp = ph * K * np.exp(GC - Gc)
        o[sl] = (tau * gam * Q) @ S + np.tril(Ap) @ Rp
        S = np.exp(GC)[:, None] * S + Kp.T @ Rp
    return o, S, n_range


# ---------------------------------------------------------------------------

def _seq(ins, b, h):
    one = {n: ins[n][b, :, h] for n in ("q", "k", "v", "g", "omega", "r")}
    dk, dv = ins["dk"], ins["dv"]
    one["S0"] = np.zeros((dk, dv)) if ins["S0"] is None else ins["S0"][b, h]
    P = dk if ins["variant"] == "diag" else 1
    one["p0"] = np.ones(P) if ins["p0"] is None else np.atleast_1d(ins["p0"][b, h])
    return one


def _decay(ins, kind, rng):
    g = ins["g"]
    if kind == "e-2":
        g = np.full_like(g, -2.0)
    elif kind == "e-3":
        g = np.full_like(g, -3.0)
    elif kind == "mixed":  # strong decay in some channels of every other 64-token chunk
        g = g.copy()
        for c0 in range(0, g.shape[1], 128):
            ch = rng.permutation(g.shape[-1])[: g.shape[-1] // 2]
            g[:, c0:c0 + 64, :, ch] = -3.5
    ins = dict(ins)
    ins["g"] = g
    return ins


CASES = [
    # variant, per-channel decay, T, dk, dv, C_g, C_m
    ("diag", True, 200, 32, 16, 256, 64),
    ("diag", True, 200, 32, 16, 64, 32),
    ("diag", True, 131, 16, 24, 40, 64),
    ("iso", False, 200, 32, 16, 256, 64),
    ("iso", True, 150, 16, 32, 64, 32),
]


@pytest.mark.parametrize("case", CASES, ids=lambda c: "-".join(map(str, c)))
def test_chunked_form_equals_token_loop(case):
    variant, pc, T, dk, dv, Cg, Cm = case
    ins = make_inputs(variant, 2, T, 2, dk, dv, dtype="f32", seed=11, per_channel_decay=pc,
                      s0_std=0.3, p0_range=(0.5, 2.0))
    mu, tau = 0.7 * dk, dk ** -0.5
    ref = oracle.fwd(variant, *[ins[n] for n in ("q", "k", "v", "g", "omega", "r")],
                     ins["S0"], ins["p0"], mu=mu, scale=tau, trace=True)
    for b in range(2):
        for h in range(2):
            x = _seq(ins, b, h)
            kappa, phat, pT = gain_chunked(variant, x["k"], x["g"], x["omega"], x["r"], x["p0"],
                                           mu, Cg)
            assert _rel(kappa, ref["kappa"][b, :, h]) <= TOL
            assert _rel(pT, np.atleast_1d(ref["pT"][b, h])) <= TOL
            G = x["g"] if x["g"].ndim == 2 else np.repeat(x["g"][:, None], dk, axis=1)
            o, ST = memory_chunked(x["q"], x["k"], x["v"], G, kappa, x["S0"], tau, Cm)
            assert _rel(o, ref["o"][b, :, h]) <= TOL
            assert _rel(ST, ref["ST"][b, h]) <= TOL


@pytest.mark.parametrize("kind", ["workload", "e-2", "e-3", "mixed"])
def test_diagonal_forward_order_equals_token_loop(kind):
    T, dk, dv = 300, 32, 16
    ins = _decay(make_inputs("diag", 1, T, 2, dk, dv, dtype="f32", seed=7, s0_std=0.05,
                             p0_range=(0.5, 2.0)), kind, np.random.default_rng(5))
    tau = dk ** -0.5
    ref = oracle.fwd("diag", *[ins[n] for n in ("q", "k", "v", "g", "omega", "r")],
                     ins["S0"], ins["p0"], scale=tau, trace=True)
    n_range = 0
    for h in range(2):
        x = _seq(ins, 0, h)
        o, ST, nr = memory_kernel_order(x["q"], x["k"], x["v"], x["g"], ref["phat"][0, :, h],
                                        x["r"], x["S0"], tau)
        n_range += nr
        assert _rel(o, ref["o"][0, :, h]) <= TOL
        assert _rel(ST, ref["ST"][0, h]) <= TOL
    # the direct form is taken by the chunks whose G_C < -160 in some channel:
    # none at the workload's decay or at alpha = e^-2 (G_C = -128); at e^-3 the
    # four full chunks of each head (G_C = -192), not the 44-token tail
    # (G_C = -132); with the mixed decays the full chunks at tokens 0 and 128
    assert n_range == {"workload": 0, "e-2": 0, "e-3": 8, "mixed": 4}[kind]


def test_solve_form_is_the_paper_inverse():
    """A = diag(s) L^-1 with L = diag(s) + strict_lower(T') equals (I + T)^-1 for
    T = strict_lower(T') diag(1/s): the kernel's solve is the paper's matrix."""
    rng = np.random.default_rng(3)
    C = 64
    Tp = rng.standard_normal((C, C)) * 0.3
    s = rng.uniform(0.5, 3.0, C)
    np.fill_diagonal(Tp, s - 0.2)       # diag(T') = s - r with r = 0.2
    A_kernel = np.diag(s) @ np.linalg.inv(np.diag(s) + np.tril(Tp, -1))
    A_paper = np.linalg.inv(np.eye(C) + np.tril(Tp, -1) @ np.diag(1.0 / s))
    assert np.max(np.abs(A_kernel - A_paper)) <= 1e-10 * np.max(np.abs(A_paper))


# ---------------------------------------------------------------------------
# the chunk adjoint the fused backward forms (the paper gives no backward)

def gain_forward(variant, k, g, omega, r, p0, mu):
    """Per-token quantities of the gain recursion (Prop. 3 / Prop. 5), token by
    token: the pre-write variance phat, the uncertainty before and after each
    token, kappa and the scalars the adjoint needs."""
    T, dk = k.shape
    alpha = np.exp(g)
    n2 = np.sum(k * k, axis=1)
    if variant == "diag":
        a, u, w = alpha * alpha, mu * k * k / r[:, None], omega
    else:
        a2 = alpha * alpha
        a = (np.mean(a2, axis=1) if g.ndim == 2 else a2)[:, None]
        u, w = (mu * n2 / (dk * r))[:, None], omega[:, None]
    p = np.broadcast_to(p0, (a.shape[1],)).astype(np.float64)
    prev, phat, post = np.empty_like(a), np.empty_like(a), np.empty_like(a)
    for t in range(T):
        prev[t] = p
        phat[t] = a[t] * p + w[t]
        p = phat[t] / (1.0 + u[t] * phat[t])
        post[t] = p
    if variant == "diag":
        s = r + np.sum(phat * k * k, axis=1)
        kappa = phat * k / s[:, None]
    else:
        s = r + phat[:, 0] * n2                       # beta = bhat / s
        kappa = (phat[:, 0] / s)[:, None] * k
    return dict(alpha=alpha, a=a, u=u, prev=prev, phat=phat, post=post, s=s, n2=n2,
                kappa=kappa)


def chunk_backward(variant, x, dO, dST, dpT, mu, tau, Cm):
    """Gradients of <dO, o> + <dS_T, S_T> + <dp_T, p_T> for one sequence: the
    memory adjoint chunk by chunk in reverse (the stages of the fused backward,
    B1-B10), then the gain adjoint token by token in reverse."""
    q, k, v, g, r = x["q"], x["k"], x["v"], x["g"], x["r"]
    T, dk = k.shape
    G = g if g.ndim == 2 else np.repeat(g[:, None], dk, axis=1)
    gn = gain_forward(variant, k, g, x["omega"], r, x["p0"], mu)
    kappa = gn["kappa"]
    starts = list(range(0, T, Cm))
    S_in, S = [], x["S0"].copy()
    for c0 in starts:                                   # forward: the memory entering each chunk
        S_in.append(S)
        _, S = memory_chunked(q[c0:c0 + Cm], k[c0:c0 + Cm], v[c0:c0 + Cm], G[c0:c0 + Cm],
                              kappa[c0:c0 + Cm], S, tau, Cm)
    dq, dk_, dv = np.zeros_like(q), np.zeros_like(k), np.zeros_like(v)
    dG, dkap = np.zeros_like(G), np.zeros_like(kappa)
    dS = dST.copy()
    for c0, Sin in zip(reversed(starts), reversed(S_in)):
        sl = slice(c0, min(c0 + Cm, T))
        C = sl.stop - sl.start
        gam = np.exp(np.cumsum(G[sl], axis=0))
        K, Kk, Q, V, dOc = k[sl], kappa[sl], q[sl], v[sl], dO[sl]
        Kbar, Kkbar, Qbar = gam * K, Kk / gam, tau * gam * Q
        A = np.linalg.inv(np.eye(C) + np.tril(Kbar @ Kkbar.T, -1))
        W = A @ Kbar
        R = A @ V - W @ Sin
        Ktail, Aqk = gam[-1] * Kkbar, np.tril(Qbar @ Kkbar.T)
        dR = Aqk.T @ dOc + Ktail @ dS                                   # B1
        dSin = gam[-1][:, None] * dS + Qbar.T @ dOc - W.T @ dR          # B2
        dAqk = np.tril(dOc @ R.T)                                       # B3
        dKtail = R @ dS.T                                               # B4
        dW = -dR @ Sin.T                                                # B5
        dv[sl] = A.T @ dR                                               # B7 (U = A V)
        dQbar = dOc @ Sin.T + dAqk @ Kkbar                              # B8
        dA = dR @ V.T + dW @ Kbar.T                                     # B6
        dT = np.tril(-A.T @ dA @ A.T, -1)                               # A = (I + T)^-1
        dKkbar = dAqk.T @ Qbar + gam[-1] * dKtail + dT.T @ Kbar         # B9
        dKbar = A.T @ dW + dT @ Kkbar                                   # B10
        dgamC = np.sum(dKtail * Kkbar, axis=0) + np.sum(dS * Sin, axis=1)
        # the scalings by Gamma, then gamma = exp(cumsum g) within the chunk
        dk_[sl] += gam * dKbar
        dkap[sl] += dKkbar / gam
        dq[sl] += tau * gam * dQbar
        dgam = K * dKbar - Kkbar * dKkbar / gam + tau * Q * dQbar
        dgam[-1] += dgamC
        dG[sl] += np.cumsum((gam * dgam)[::-1], axis=0)[::-1]
        dS = dSin
    # gain adjoint, tokens in reverse (eqs. kla-box-gain, diag-cov-update / Prop. 5)
    a, u, prev, phat, post, s = gn["a"], gn["u"], gn["prev"], gn["phat"], gn["post"], gn["s"]
    alpha, n2 = gn["alpha"], gn["n2"]
    domega = np.zeros_like(x["omega"])
    dr = np.zeros_like(r)
    dgate = np.zeros_like(G)            # d/dalpha terms of the uncertainty, as d/dg
    dp = np.broadcast_to(dpT, (a.shape[1],)).astype(np.float64)
    for t in range(T - 1, -1, -1):
        dphat = dp / (1.0 + u[t] * phat[t]) ** 2       # p = phat / (1 + u phat)
        du = -dp * post[t] ** 2
        if variant == "diag":
            dk_[t] += du * 2.0 * mu * k[t] / r[t]
            dr[t] -= np.sum(du * u[t]) / r[t]
            c = np.sum(dkap[t] * kappa[t])
            ds = -c / s[t]
            dphat += dkap[t] * k[t] / s[t] + ds * k[t] ** 2
            dk_[t] += dkap[t] * phat[t] / s[t] + 2.0 * ds * phat[t] * k[t]
            dr[t] += ds
            domega[t] = dphat
            dgate[t] += 2.0 * alpha[t] ** 2 * prev[t] * dphat
        else:
            dn2 = du[0] * mu / (dk * r[t])
            dr[t] -= du[0] * u[t, 0] / r[t]
            beta = phat[t, 0] / s[t]
            dbeta = np.dot(dkap[t], k[t])
            dk_[t] += beta * dkap[t]
            dphat = dphat + dbeta * r[t] / s[t] ** 2
            dr[t] -= dbeta * beta / s[t]
            dn2 -= dbeta * beta ** 2
            dk_[t] += 2.0 * k[t] * dn2
            domega[t] = dphat[0]
            da = prev[t, 0] * dphat[0]                  # a = mean alpha^2 (or alpha^2)
            if g.ndim == 2:
                dgate[t] += da * 2.0 * alpha[t] ** 2 / dk
            else:
                dgate[t] += da * 2.0 * alpha[t] ** 2
        dp = a[t] * dphat
    if g.ndim == 2:
        dg = dG + dgate
    else:  # one decay per head: every channel's log-decay is g_t
        dg = np.sum(dG, axis=1) + dgate[:, 0]
    return dict(dq=dq, dk=dk_, dv=dv, dg=dg, domega=domega, dr=dr, dS0=dS, dp0=dp)


BWD_CASES = [
    # variant, per-channel decay, T, dk, dv, C_m
    ("diag", True, 150, 16, 24, 64),
    ("diag", True, 97, 32, 16, 32),
    ("iso", True, 130, 16, 16, 64),
    ("iso", False, 100, 32, 16, 32),
]


@pytest.mark.parametrize("case", BWD_CASES, ids=lambda c: "-".join(map(str, c)))
def test_chunk_adjoint_equals_token_loop_adjoint(case):
    """The chunk adjoint of the fused backward (B1-B10 and the scalings by
    Gamma), followed by the gain adjoint, gives the oracle's gradients (which
    are pinned to finite differences) with nonzero dS_T and dp_T."""
    variant, pc, T, dk, dv, Cm = case
    ins = make_inputs(variant, 1, T, 2, dk, dv, dtype="f32", seed=21, per_channel_decay=pc,
                      s0_std=0.3, p0_range=(0.5, 2.0), with_grad=True)
    rng = np.random.default_rng(4)
    P = dk if variant == "diag" else 1
    dST = rng.standard_normal((1, 2, dk, dv))
    dpT = rng.standard_normal((1, 2, P) if variant == "diag" else (1, 2))
    mu, tau = 0.7 * dk, dk ** -0.5
    ref = oracle.bwd(variant, *[ins[n] for n in ("q", "k", "v", "g", "omega", "r")],
                     ins["S0"], ins["p0"], ins["dO"], dST, dpT, mu=mu, scale=tau)
    for h in range(2):
        x = _seq(ins, 0, h)
        got = chunk_backward(variant, x, ins["dO"][0, :, h], dST[0, h],
                             np.atleast_1d(dpT[0, h]), mu, tau, Cm)
        for n in ("dq", "dk", "dv", "dg", "domega", "dr", "dS0", "dp0"):
            want = ref[n][0, :, h] if ref[n].ndim >= 3 and n not in ("dS0", "dp0") else ref[n][0, h]
            assert _rel(got[n].reshape(np.shape(want)), np.asarray(want)) <= TOL, n


# ---------------------------------------------------------------------------
# the sequence-parallel forward: segments joined exactly

def token_matrices(variant, k, g, omega, r, mu):
    """The Moebius matrices M_t [T, P, 2, 2] of the uncertainty update."""
    T, dk = k.shape
    if variant == "diag":
        a, u, w = np.exp(2.0 * g), mu * k * k / r[:, None], omega
    else:
        a = (np.mean(np.exp(2.0 * g), axis=1) if g.ndim == 2 else np.exp(2.0 * g))[:, None]
        u, w = (mu * np.sum(k * k, axis=1) / (dk * r))[:, None], omega[:, None]
    M = np.empty((T,) + a.shape[1:] + (2, 2))
    M[..., 0, 0], M[..., 0, 1], M[..., 1, 0], M[..., 1, 1] = a, w, u * a, 1.0 + u * w
    return M


def segmented_forward(variant, x, mu, tau, P, C=64, join=True):
    """o, S_T, p_T of one sequence cut into P segments of whole chunks, as the
    sequence-parallel forward joins them:
      * level 1: each chunk's Moebius summary, and each segment's product of its
        chunk summaries (neither depends on p_0);
      * level 2: the exclusive scan of the segment products from z_0 = [p_0, 1]
        gives the uncertainty entering each segment, from which every segment
        replays its gains;
      * per segment, with the gains fixed: the memory from S_in = 0 with v (exit
        Sv_j, outputs o_v) and the transition Phi_j from S_in = I with v = 0
        (outputs o_Phi = tau Phi_t^T q_t);
      * the join S_in(j+1) = Phi_j S_in(j) + Sv_j, o_t = o_v,t + S_in(j)^T o_Phi,t.
    ``join`` = False runs every segment on its own from S = 0 and p = 1."""
    q, k, v, g, omega, r = (x[n] for n in ("q", "k", "v", "g", "omega", "r"))
    T, dk = k.shape
    nc = -(-T // C)
    assert nc % P == 0
    seg = (nc // P) * C
    segs = [slice(j * seg, min((j + 1) * seg, T)) for j in range(P)]
    G = g if g.ndim == 2 else np.repeat(g[:, None], dk, axis=1)
    M = token_matrices(variant, k, g, omega, r, mu)
    Pn = M.shape[1]
    # level 1: chunk summaries, then segment products (later chunks on the left)
    seg_prod = []
    for sl in segs:
        prod = np.broadcast_to(np.eye(2), (Pn, 2, 2)).copy()
        for c0 in range(sl.start, sl.stop, C):
            summ = np.broadcast_to(np.eye(2), (Pn, 2, 2)).copy()
            for t in range(c0, min(c0 + C, T)):
                summ = _renorm(np.einsum("pij,pjk->pik", M[t], summ))
            prod = _renorm(np.einsum("pij,pjk->pik", summ, prod))
        seg_prod.append(prod)
    # level 2: exclusive scan of the segment products from z_0
    p0 = x["p0"] if join else np.ones_like(x["p0"])
    z = np.stack([np.broadcast_to(p0, (Pn,)), np.ones(Pn)], axis=1)
    p_in = []
    for prod in seg_prod:
        p_in.append(z[:, 0] / z[:, 1] if join else np.ones(Pn))
        z = _renorm(np.einsum("pij,pj->pi", prod, z))
    p_T = z[:, 0] / z[:, 1]
    kappa = np.empty_like(k)
    for sl, pj in zip(segs, p_in):
        kappa[sl], _, _ = gain_chunked(variant, k[sl], g[sl], omega[sl], r[sl], pj, mu, C)
    # per segment: the memory from 0 and the transition from I
    o_v, o_phi, Sv, Phi = np.empty((T, v.shape[1])), np.empty((T, dk)), [], []
    for sl in segs:
        S, F = np.zeros((dk, v.shape[1])), np.eye(dk)
        for t in range(sl.start, sl.stop):
            a = np.exp(G[t])
            Sh, Fh = a[:, None] * S, a[:, None] * F
            S = Sh + np.outer(kappa[t], v[t] - Sh.T @ k[t])
            F = Fh - np.outer(kappa[t], Fh.T @ k[t])
            o_v[t], o_phi[t] = tau * S.T @ q[t], tau * F.T @ q[t]
        Sv.append(S)
        Phi.append(F)
    if not join:
        return o_v, None, None
    S_in = x["S0"]
    o = np.empty_like(o_v)
    for sl, Sj, Fj in zip(segs, Sv, Phi):
        o[sl] = o_v[sl] + o_phi[sl] @ S_in
        S_in = Fj @ S_in + Sj
    return o, S_in, p_T


@pytest.mark.parametrize("variant,pc", [("diag", True), ("iso", False), ("iso", True)])
def test_sequence_parallel_join_equals_token_loop(variant, pc):
    """The join of the sequence-parallel forward is exact: with decays near 1, so
    that memory and uncertainty carry across whole segments, the joined result
    equals the token loop to 1e-9 in fp64, and differs from the segments run on
    their own by far more than rounding."""
    T, dk, dv, P = 512, 16, 8, 4
    ins = make_inputs(variant, 1, T, 1, dk, dv, dtype="f32", seed=17, per_channel_decay=pc,
                      s0_std=0.5, p0_range=(0.5, 2.0))
    ins["g"] = ins["g"] * 0.02          # alpha ~ 0.997: long memory
    mu, tau = float(dk), dk ** -0.5
    ref = oracle.fwd(variant, *[ins[n] for n in ("q", "k", "v", "g", "omega", "r")],
                     ins["S0"], ins["p0"], mu=mu, scale=tau)
    x = _seq(ins, 0, 0)
    o, ST, pT = segmented_forward(variant, x, mu, tau, P)
    assert _rel(o, ref["o"][0, :, 0]) <= TOL
    assert _rel(ST, ref["ST"][0, 0]) <= TOL
    assert _rel(pT, np.atleast_1d(ref["pT"][0, 0])) <= TOL
    alone, _, _ = segmented_forward(variant, x, mu, tau, P, join=False)
    assert _rel(alone, ref["o"][0, :, 0]) > 1e-2
