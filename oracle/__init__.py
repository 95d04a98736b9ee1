"""fp64 CPU oracle for the Kalman Delta Network token mixers (ctypes binding).

TEST INFRASTRUCTURE ONLY.  Only ``tests/``, ``__graft_entry__.smoke()`` and the
CPU-baseline leg of ``bench.py`` may import this package.  The product library
(``paper_2609_07816_gb300``) never imports it and shares no code with it.

The C source (``kdn_oracle.c``) is a token-by-token float64 transcription of
Prop. 3 (Diagonal KDN) and Prop. 5 (Isotropic KDN) plus the hand-derived
adjoint of that token loop.  This module only marshals numpy arrays.

Array layouts (all float64, C-contiguous):
  q, k [B,T,H,dk]; v [B,T,H,dv]; r [B,T,H];
  diag: g, omega [B,T,H,dk]; iso: omega [B,T,H], g [B,T,H,dk] or [B,T,H];
  S0 [B,H,dk,dv]; p0 diag [B,H,dk], iso [B,H].
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "kdn_oracle.c")
_LIB_PATH = os.path.join(_HERE, "libkdn_oracle.so")
_lib = None
_lock = threading.Lock()


def build(force: bool = False) -> str:
    """Compile the oracle into ``oracle/libkdn_oracle.so`` with gcc (no fast-math)."""
    if (not force and os.path.exists(_LIB_PATH)
            and os.path.getmtime(_LIB_PATH) >= os.path.getmtime(_SRC)):
        return _LIB_PATH
    tmp = _LIB_PATH + f".tmp{os.getpid()}"
    cmd = ["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-fno-fast-math",
           "-ffp-contract=off", "-o", tmp, _SRC, "-lm", "-lpthread"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _load():
    global _lib
    with _lock:
        if _lib is None:
            build()
            lib = ctypes.CDLL(_LIB_PATH)
            P = ctypes.c_void_p
            I = ctypes.c_int
            D = ctypes.c_double
            lib.kdn_oracle_fwd.argtypes = [I, I, I, I, I, I, D, D, I] + [P] * 15 + [I]
            lib.kdn_oracle_fwd.restype = I
            lib.kdn_oracle_bwd.argtypes = [I, I, I, I, I, I, D, D, I] + [P] * 21 + [I]
            lib.kdn_oracle_bwd.restype = I
            _lib = lib
    return _lib


def _ptr(a):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


def _f64(a):
    if a is None:
        return None
    return np.ascontiguousarray(a, dtype=np.float64)


def _defaults(dk, mu, scale):
    mu = float(dk) if (mu is None or mu <= 0) else float(mu)
    scale = 1.0 / np.sqrt(dk) if scale is None else float(scale)
    return mu, scale


def _variant(name):
    if name in ("diag", 0):
        return 0
    if name in ("iso", 1):
        return 1
    raise ValueError(f"unknown variant {name!r}")


def _softplus(x):
    return np.logaddexp(0.0, x)


def _sigmoid(x):
    return np.exp(-np.logaddexp(0.0, -x))


def gates_from_logits(x, y, z, r_min):
    """The layer's gate parameterisation (eq. kla-box-parameterization, r_min of
    Sec. 5): alpha = sigmoid(x), omega = softplus(y), r = r_min + softplus(z).
    Returns (g = log alpha, omega, r) in float64."""
    x, y, z = map(_f64, (x, y, z))
    return -_softplus(-x), _softplus(y), r_min + _softplus(z)


def _check_gates(gates):
    if gates not in ("post", "logits"):
        raise ValueError(gates)


def fwd(variant, q, k, v, g, omega, r, S0=None, p0=None, *, mu=None, scale=None,
        bhat=None, trace=False, threads=0, gates="post", r_min=0.01):
    """Forward over all tokens.  Returns dict(o, ST, pT[, kappa, phat, p], threads).

    ``bhat`` (isotropic only) switches to the surrogate mode of
    eq. fixed-gain-approx: the predicted variance is taken from ``bhat`` [B,T,H]
    instead of being tracked.  ``gates="logits"``: g, omega, r are the logits of
    the layer's parameterisation (``gates_from_logits``).
    """
    _check_gates(gates)
    if gates == "logits":
        g, omega, r = gates_from_logits(g, omega, r, r_min)
    lib = _load()
    vid = _variant(variant)
    q, k, v, g, omega, r = map(_f64, (q, k, v, g, omega, r))
    S0, p0, bhat = _f64(S0), _f64(p0), _f64(bhat)
    B, T, H, dk = q.shape
    dv = v.shape[-1]
    mu, scale = _defaults(dk, mu, scale)
    per_channel = int(g.ndim == 4)
    np_ = dk if vid == 0 else 1
    o = np.zeros((B, T, H, dv))
    ST = np.zeros((B, H, dk, dv))
    pT = np.zeros((B, H, dk) if vid == 0 else (B, H))
    kap = np.zeros((B, T, H, dk)) if trace else None
    phat = np.zeros((B, T, H, np_)) if trace else None
    pt = np.zeros((B, T, H, np_)) if trace else None
    n = lib.kdn_oracle_fwd(vid, B, T, H, dk, dv, mu, scale, per_channel,
                           _ptr(q), _ptr(k), _ptr(v), _ptr(g), _ptr(omega), _ptr(r),
                           _ptr(S0), _ptr(p0), _ptr(bhat), _ptr(o), _ptr(ST), _ptr(pT),
                           _ptr(kap), _ptr(phat), _ptr(pt), int(threads))
    if n < 0:
        raise ValueError("oracle rejected the arguments")
    out = dict(o=o, ST=ST, pT=pT, threads=n)
    if trace:
        out.update(kappa=kap, phat=phat if vid == 0 else phat[..., 0],
                   p=pt if vid == 0 else pt[..., 0])
    return out


def bwd(variant, q, k, v, g, omega, r, S0, p0, dO, dST=None, dpT=None, *, mu=None,
        scale=None, bhat=None, threads=0, gates="post", r_min=0.01):
    """Gradients of <dO, o> + <dST, ST> + <dpT, pT> with respect to every input,
    and ``dmu`` [B,H]: with respect to the information scale mu of each sequence.

    ``gates="logits"``: g, omega, r are logits, and dg, domega, dr are the
    gradients with respect to them (chain rule through ``gates_from_logits``:
    d log alpha / dx = sigmoid(-x), d omega / dy = sigmoid(y), d r / dz = sigmoid(z)).
    """
    _check_gates(gates)
    if gates == "logits":
        x, y, z = map(_f64, (g, omega, r))
        g, omega, r = gates_from_logits(x, y, z, r_min)
        out = bwd(variant, q, k, v, g, omega, r, S0, p0, dO, dST, dpT, mu=mu, scale=scale,
                  bhat=bhat, threads=threads)
        out["dg"] = out["dg"] * _sigmoid(-x)
        out["domega"] = out["domega"] * _sigmoid(y)
        out["dr"] = out["dr"] * _sigmoid(z)
        return out
    lib = _load()
    vid = _variant(variant)
    q, k, v, g, omega, r, dO = map(_f64, (q, k, v, g, omega, r, dO))
    S0, p0, dST, dpT, bhat = map(_f64, (S0, p0, dST, dpT, bhat))
    B, T, H, dk = q.shape
    dv = v.shape[-1]
    mu, scale = _defaults(dk, mu, scale)
    per_channel = int(g.ndim == 4)
    out = dict(dq=np.zeros_like(q), dk=np.zeros_like(k), dv=np.zeros_like(v),
               dg=np.zeros_like(g), domega=np.zeros_like(omega), dr=np.zeros_like(r),
               dS0=np.zeros((B, H, dk, dv)),
               dp0=np.zeros((B, H, dk) if vid == 0 else (B, H)), dmu=np.zeros((B, H)))
    n = lib.kdn_oracle_bwd(vid, B, T, H, dk, dv, mu, scale, per_channel,
                           _ptr(q), _ptr(k), _ptr(v), _ptr(g), _ptr(omega), _ptr(r),
                           _ptr(S0), _ptr(p0), _ptr(bhat), _ptr(dO), _ptr(dST), _ptr(dpT),
                           _ptr(out["dq"]), _ptr(out["dk"]), _ptr(out["dv"]),
                           _ptr(out["dg"]), _ptr(out["domega"]), _ptr(out["dr"]),
                           _ptr(out["dS0"]), _ptr(out["dp0"]), _ptr(out["dmu"]), int(threads))
    if n < 0:
        raise ValueError("oracle rejected the arguments")
    out["threads"] = n
    return out


def decode_step(variant, q, k, v, g, omega, r, S, p, *, mu=None, scale=None, gates="post",
                r_min=0.01):
    """One token of the recurrence on a given state (T = 1 of ``fwd``).

    Inputs are per-step arrays without the T axis: q, k [B,H,dk], v [B,H,dv],
    r [B,H], gates [B,H,dk] or [B,H].  Returns (o [B,H,dv], S_new, p_new).
    """
    ins = [None if a is None else np.asarray(a, dtype=np.float64)[:, None]
           for a in (q, k, v, g, omega, r)]
    res = fwd(variant, *ins, S0=S, p0=p, mu=mu, scale=scale, gates=gates, r_min=r_min)
    return res["o"][:, 0], res["ST"], res["pT"]
