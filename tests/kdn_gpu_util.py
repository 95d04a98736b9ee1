"""Helpers shared by the GPU parity tests: move generator inputs to the device
and compare a GPU tensor with the oracle under the tolerance rule

    max |gpu - oracle| <= tol * RMS(oracle)

with tol = 1e-4 for float32 activations and 2e-2 for bfloat16 activations
(float32 state and accumulation in both cases)."""
import numpy as np
import torch

TORCH_DT = {"f32": torch.float32, "bf16": torch.bfloat16}
TOL = {"f32": 1e-4, "bf16": 2e-2}
GATE_NAMES = ("q", "k", "v", "g", "omega", "r")


def to_dev(ins, device="cuda"):
    dt = TORCH_DT[ins["dtype"]]
    out = {n: torch.tensor(ins[n], dtype=dt, device=device) for n in GATE_NAMES}
    for n in ("S0", "p0"):
        out[n] = None if ins.get(n) is None else torch.tensor(ins[n], dtype=torch.float32,
                                                               device=device)
    if ins.get("dO") is not None:
        out["dO"] = torch.tensor(ins["dO"], dtype=dt, device=device)
    return out


def to_np(x):
    return x.detach().float().cpu().double().numpy()


def err_ratio(gpu, ref):
    g = to_np(gpu) if torch.is_tensor(gpu) else np.asarray(gpu, dtype=np.float64)
    rms = float(np.sqrt(np.mean(np.square(ref)))) if ref.size else 0.0
    if not np.all(np.isfinite(g)):
        return float("inf")
    err = float(np.max(np.abs(g - ref))) if ref.size else 0.0
    return err / rms if rms > 0 else (0.0 if err == 0 else float("inf"))


def check(name, gpu, ref, dtype, report=None):
    r = err_ratio(gpu, ref)
    if report is not None:
        report[name] = r
    assert r <= TOL[dtype], f"{name}: max|err|/RMS = {r:.3e} > {TOL[dtype]}"
    return r


def head_slice(ins, b, h):
    """Inputs of one (b, h) sequence as a B=1, H=1 problem (oracle side)."""
    out = dict(ins)
    for n in GATE_NAMES + ("dO",):
        if ins.get(n) is not None:
            out[n] = ins[n][b:b + 1, :, h:h + 1]
    for n in ("S0", "p0"):
        if ins.get(n) is not None:
            out[n] = ins[n][b:b + 1, h:h + 1]
    return out


def check_stored_bf16(name, gpu, ref, report=None):
    """bfloat16 outputs: the float32 result must meet the bf16-input rule before
    its final rounding to the stored dtype, so allow that one rounding on top:
    |gpu - ref| <= 2e-2 * RMS(ref) + 2^-8 |ref|  (2^-8 = bf16 unit roundoff)."""
    g = to_np(gpu)
    rms = float(np.sqrt(np.mean(np.square(ref))))
    excess = np.abs(g - ref) - 2.0 ** -8 * np.abs(ref)
    r = float(np.max(excess)) / rms if rms > 0 else 0.0
    if report is not None:
        report[name] = r
    assert np.all(np.isfinite(g)) and r <= TOL["bf16"], f"{name}: {r:.3e}"
    return r
