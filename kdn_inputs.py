"""Seeded synthetic inputs for the KDN token mixers.

This module is shared by the oracle tests, the CUDA parity tests and the
benchmark.  It holds no arithmetic of the method itself: it only draws random
numbers, normalises keys/queries, applies the input activations the paper
places *before* the layer (log-sigmoid decay, softplus noises; Prop. 3
parameterisation eq. kla-box-parameterization) and rounds to the storage dtype.

Recipe (matches the measured workloads):
  * q, k ~ N(0, 1), then L2-normalised over d_k for every (b, t, h);
  * v ~ N(0, 1);
  * decay alpha = sigmoid(x), x ~ N(2, 1), passed as g = log(alpha) <= 0;
    per channel [B,T,H,dk] (Diagonal KDN, Isotropic KDN per-channel mode) or
    one scalar per head [B,T,H] (Isotropic KDN scalar mode);
  * process noise omega = softplus(N(0, 1)) per channel (diag) / per head (iso);
  * observation noise r = softplus(N(0, 1)) per head, no r_min added;
  * initial memory S_0 = 0 or N(0, s0_std^2); initial uncertainty 1 or U(lo, hi);
  * upstream gradient dO ~ N(0, 1).
Draw order is fixed: q, k, v, x_decay, x_omega, x_r, S_0, p_0, dO.  Values are
generated in float64, rounded once to the storage dtype (bf16 by round-to-
nearest-even through float32, or float32), and returned as float64 arrays that
hold exactly the rounded values, so the oracle and the GPU see identical
inputs.
"""
from __future__ import annotations

import numpy as np

DTYPES = ("f32", "bf16")


def round_to(x: np.ndarray, dtype: str) -> np.ndarray:
    """Round float64 values to ``dtype`` and return them as float64."""
    x32 = np.asarray(x, dtype=np.float64).astype(np.float32)
    if dtype == "f32":
        return x32.astype(np.float64)
    if dtype != "bf16":
        raise ValueError(dtype)
    u = x32.view(np.uint32).astype(np.uint64)
    u = (u + 0x7FFF + ((u >> 16) & 1)) >> 16
    back = (u.astype(np.uint32) << 16).view(np.float32)
    return back.astype(np.float64)


def _l2n(x):
    return x / np.sqrt(np.sum(x * x, axis=-1, keepdims=True))


def _softplus(x):
    return np.logaddexp(0.0, x)


def _log_sigmoid(x):
    return -np.logaddexp(0.0, -x)


def make_inputs(variant: str, B: int, T: int, H: int, dk: int, dv: int, *,
                dtype: str = "bf16", seed: int = 0, per_channel_decay: bool | None = None,
                s0_std: float = 0.0, p0_range: tuple | None = None,
                with_grad: bool = False) -> dict:
    """Draw one batch.  Returns a dict of float64 arrays plus metadata.

    ``variant`` is "diag" or "iso".  ``per_channel_decay`` defaults to True for
    diag and False for iso.
    """
    if variant not in ("diag", "iso"):
        raise ValueError(variant)
    if per_channel_decay is None:
        per_channel_decay = variant == "diag"
    if variant == "diag" and not per_channel_decay:
        raise ValueError("Diagonal KDN has per-channel decay")
    rng = np.random.Generator(np.random.PCG64(seed))
    q = _l2n(rng.standard_normal((B, T, H, dk)))
    k = _l2n(rng.standard_normal((B, T, H, dk)))
    v = rng.standard_normal((B, T, H, dv))
    gshape = (B, T, H, dk) if per_channel_decay else (B, T, H)
    g = _log_sigmoid(rng.normal(2.0, 1.0, size=gshape))
    wshape = (B, T, H, dk) if variant == "diag" else (B, T, H)
    omega = _softplus(rng.standard_normal(wshape))
    r = _softplus(rng.standard_normal((B, T, H)))
    S0 = rng.normal(0.0, s0_std, size=(B, H, dk, dv)) if s0_std > 0 else None
    pshape = (B, H, dk) if variant == "diag" else (B, H)
    p0 = rng.uniform(p0_range[0], p0_range[1], size=pshape) if p0_range else None
    dO = rng.standard_normal((B, T, H, dv)) if with_grad else None

    out = dict(variant=variant, dtype=dtype, B=B, T=T, H=H, dk=dk, dv=dv,
               per_channel_decay=bool(per_channel_decay))
    for name, arr in (("q", q), ("k", k), ("v", v), ("g", g), ("omega", omega), ("r", r)):
        out[name] = round_to(arr, dtype)
    # recurrent state is always float32 in the library
    out["S0"] = None if S0 is None else round_to(S0, "f32")
    out["p0"] = None if p0 is None else round_to(p0, "f32")
    out["dO"] = None if dO is None else round_to(dO, dtype)
    return out


def make_decode_inputs(variant: str, B: int, H: int, dk: int, dv: int, steps: int, *,
                       dtype: str = "bf16", seed: int = 0, s_std: float = 0.02,
                       p_range: tuple = (0.1, 2.0), per_channel_decay: bool | None = None) -> dict:
    """Initial state plus ``steps`` fresh per-step inputs for the decode step.

    Draw order: S, p, then for every step (q, k, v, x_decay, x_omega, x_r).
    Per-step arrays are stacked on a leading ``steps`` axis with shapes
    q, k [steps,B,H,dk], v [steps,B,H,dv], r [steps,B,H], gates [steps,B,H,dk]
    or [steps,B,H].
    """
    if per_channel_decay is None:
        per_channel_decay = variant == "diag"
    rng = np.random.Generator(np.random.PCG64(seed))
    S = rng.normal(0.0, s_std, size=(B, H, dk, dv))
    pshape = (B, H, dk) if variant == "diag" else (B, H)
    p = rng.uniform(p_range[0], p_range[1], size=pshape)
    cols = {n: [] for n in ("q", "k", "v", "g", "omega", "r")}
    for _ in range(steps):
        one = draw_decode_step(rng, variant, B, H, dk, dv, per_channel_decay=per_channel_decay)
        for n in cols:
            cols[n].append(one[n])
    out = dict(variant=variant, dtype=dtype, B=B, H=H, dk=dk, dv=dv, steps=steps,
               per_channel_decay=bool(per_channel_decay),
               S=round_to(S, "f32"), p=round_to(p, "f32"))
    for n, lst in cols.items():
        out[n] = round_to(np.stack(lst), dtype)
    return out


def draw_decode_step(rng, variant: str, B: int, H: int, dk: int, dv: int, *,
                     per_channel_decay: bool, dtype: str | None = None) -> dict:
    """One decode token's inputs, drawn from ``rng`` in the order q, k, v,
    x_decay, x_omega, x_r; rounded to ``dtype`` when one is given.  Long decode
    runs draw step by step so that no [steps, B, H, d] float64 array is held."""
    gshape = (B, H, dk) if per_channel_decay else (B, H)
    wshape = (B, H, dk) if variant == "diag" else (B, H)
    one = {"q": _l2n(rng.standard_normal((B, H, dk))),
           "k": _l2n(rng.standard_normal((B, H, dk))),
           "v": rng.standard_normal((B, H, dv)),
           "g": _log_sigmoid(rng.normal(2.0, 1.0, size=gshape)),
           "omega": _softplus(rng.standard_normal(wshape)),
           "r": _softplus(rng.standard_normal((B, H)))}
    if dtype is not None:
        one = {n: round_to(x, dtype) for n, x in one.items()}
    return one
