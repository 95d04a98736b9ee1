"""GPU parity with logit gates (KDN_GATES_LOGITS): alpha = sigmoid(x),
omega = softplus(y), r = r_min + softplus(z) applied inside the kernels, and the
backward returning gradients with respect to x, y, z; against the oracle in the
same mode, on every path (fused and general forward and backward, the training
pair, the sequence-parallel forward, decode) and with ragged tails (the padded
tokens of the last chunk must stay identity updates)."""
import numpy as np
import pytest
import torch

import oracle
from kdn_inputs import make_decode_inputs, make_inputs, round_to
from kdn_gpu_util import check, to_dev

pytestmark = pytest.mark.gpu

R_MIN = 0.01
NAMES = ("q", "k", "v", "g", "omega", "r")


@pytest.fixture(scope="module")
def kdn():
    from paper_2609_07816_gb300 import build
    build.build()
    import paper_2609_07816_gb300 as m
    torch.cuda.init()
    return m


def _logits(ins, dtype, seed):
    """Replace the gates by logits shaped like the workload's: x ~ N(2, 1) (so that
    sigmoid(x) is the decay distribution of the configs), y, z ~ N(0, 1)."""
    rng = np.random.default_rng(seed)
    ins = dict(ins)
    ins["g"] = round_to(rng.normal(2.0, 1.0, ins["g"].shape), dtype)
    ins["omega"] = round_to(rng.normal(0.0, 1.0, ins["omega"].shape), dtype)
    ins["r"] = round_to(rng.normal(0.0, 1.0, ins["r"].shape), dtype)
    return ins


def _fns(kdn, variant):
    if variant == "diag":
        return kdn.kdn_diag_fwd, kdn.kdn_diag_bwd, kdn.kdn_diag_fwd_save, kdn.kdn_diag_bwd_saved
    return kdn.kdn_iso_fwd, kdn.kdn_iso_bwd, kdn.kdn_iso_fwd_save, kdn.kdn_iso_bwd_saved


CASES = [
    # variant, per-channel decay, dtype, B, T, H, dk, dv   (path)
    ("diag", True, "bf16", 2, 150, 2, 128, 128),   # fused, ragged tail
    ("iso", False, "bf16", 1, 130, 2, 128, 128),   # fused, scalar decay
    ("iso", True, "bf16", 1, 100, 2, 128, 128),    # fused, per-channel decay
    ("diag", True, "f32", 1, 75, 2, 32, 32),       # general kernels
    ("iso", False, "f32", 2, 50, 2, 64, 32),       # general kernels
    ("iso", True, "f32", 1, 45, 1, 32, 64),        # general kernels
]


@pytest.mark.parametrize("case", CASES, ids=lambda c: "-".join(map(str, c)))
def test_logit_gates_forward_backward(kdn, case):
    variant, pc, dt, B, T, H, dk, dv = case
    ins = _logits(make_inputs(variant, B, T, H, dk, dv, dtype=dt, seed=T + dk, s0_std=0.05,
                              p0_range=(0.5, 2.0), per_channel_decay=pc, with_grad=True), dt, 7)
    kw = dict(gates=kdn.KDN_GATES_LOGITS, r_min=R_MIN)
    fwd, bwd, _, _ = _fns(kdn, variant)
    d = to_dev(ins)
    x = [d[n] for n in NAMES]
    o, ST, pT = fwd(*x, d["S0"], d["p0"], **kw)
    grads = bwd(*x, d["S0"], d["p0"], d["dO"], **kw)
    torch.cuda.synchronize()
    ref = oracle.fwd(variant, *[ins[n] for n in NAMES], ins["S0"], ins["p0"], gates="logits",
                     r_min=R_MIN)
    gref = oracle.bwd(variant, *[ins[n] for n in NAMES], ins["S0"], ins["p0"], ins["dO"],
                      gates="logits", r_min=R_MIN)
    check("o", o, ref["o"], dt)
    check("ST", ST, ref["ST"], dt)
    check("pT", pT, ref["pT"], dt)
    for n in ("dq", "dk", "dv", "dg", "domega", "dr", "dS0", "dp0", "dmu"):
        check(n, grads[n], gref[n], dt)


@pytest.mark.parametrize("variant,pc", [("diag", True), ("iso", False)])
def test_logit_gates_training_pair(kdn, variant, pc):
    """kdn_*_fwd_save / kdn_*_bwd_saved with logit gates match the oracle."""
    B, T, H = 1, 200, 2
    ins = _logits(make_inputs(variant, B, T, H, 128, 128, dtype="bf16", seed=3, s0_std=0.05,
                              p0_range=(0.5, 2.0), per_channel_decay=pc, with_grad=True),
                  "bf16", 11)
    kw = dict(gates=kdn.KDN_GATES_LOGITS, r_min=R_MIN)
    _, _, fsave, bsaved = _fns(kdn, variant)
    d = to_dev(ins)
    x = [d[n] for n in NAMES]
    o, ST, pT, saved = fsave(*x, d["S0"], d["p0"], **kw)
    grads = bsaved(*x, saved, d["dO"], **kw)
    torch.cuda.synchronize()
    ref = oracle.fwd(variant, *[ins[n] for n in NAMES], ins["S0"], ins["p0"], gates="logits",
                     r_min=R_MIN)
    # the saved-context backward has no S_0 / p_0 inputs: the cotangents of o only
    gref = oracle.bwd(variant, *[ins[n] for n in NAMES], ins["S0"], ins["p0"], ins["dO"],
                      gates="logits", r_min=R_MIN)
    check("o", o, ref["o"], "bf16")
    for n in ("dq", "dk", "dv", "dg", "domega", "dr"):
        check(n, grads[n], gref[n], "bf16")


@pytest.mark.parametrize("variant,pc", [("diag", True), ("iso", False), ("iso", True)])
def test_logit_gates_sequence_parallel_forward(kdn, variant, pc):
    """The sequence-parallel forward (gain summaries from the logits) matches the
    oracle; the decay logits x ~ N(6, 1) keep the state across segments."""
    B, T, H = 1, 2048, 2
    ins = make_inputs(variant, B, T, H, 128, 128, dtype="bf16", seed=19, s0_std=0.02,
                      p0_range=(0.5, 2.0), per_channel_decay=pc)
    ins = _logits(ins, "bf16", 23)
    rng = np.random.default_rng(29)
    ins["g"] = round_to(rng.normal(6.0, 1.0, ins["g"].shape), "bf16")
    desc = kdn.make_desc(B, T, H, 128, 128, kdn.KDN_BF16, decay_per_channel=int(pc),
                         gates=kdn.KDN_GATES_LOGITS, r_min=R_MIN)
    assert kdn.kdn_kernel_launches(desc, 0 if variant == "diag" else 1, 0) == 5
    fwd = kdn.kdn_diag_fwd if variant == "diag" else kdn.kdn_iso_fwd
    d = to_dev(ins)
    o, ST, pT = fwd(*[d[n] for n in NAMES], d["S0"], d["p0"], gates=kdn.KDN_GATES_LOGITS,
                    r_min=R_MIN)
    torch.cuda.synchronize()
    ref = oracle.fwd(variant, *[ins[n] for n in NAMES], ins["S0"], ins["p0"], gates="logits",
                     r_min=R_MIN)
    check("o", o, ref["o"], "bf16")
    check("ST", ST, ref["ST"], "bf16")
    check("pT", pT, ref["pT"], "bf16")


@pytest.mark.parametrize("variant", ["diag", "iso"])
def test_logit_gates_decode(kdn, variant):
    steps = 3
    ins = make_decode_inputs(variant, 4, 2, 128, 128, steps, dtype="bf16", seed=5)
    rng = np.random.default_rng(31)
    for n, mean in (("g", 2.0), ("omega", 0.0), ("r", 0.0)):
        ins[n] = round_to(rng.normal(mean, 1.0, ins[n].shape), "bf16")
    S = torch.tensor(ins["S"], dtype=torch.float32, device="cuda")
    p = torch.tensor(ins["p"], dtype=torch.float32, device="cuda")
    fn = kdn.kdn_diag_decode_step if variant == "diag" else kdn.kdn_iso_decode_step
    Sr, pr = ins["S"].copy(), ins["p"].copy()
    for t in range(steps):
        step = {n: torch.tensor(ins[n][t], dtype=torch.bfloat16, device="cuda") for n in NAMES}
        o = fn(*[step[n] for n in NAMES], S, p, gates=kdn.KDN_GATES_LOGITS, r_min=R_MIN)
        oref, Sr, pr = oracle.decode_step(variant, *[ins[n][t] for n in NAMES], Sr, pr,
                                          gates="logits", r_min=R_MIN)
        torch.cuda.synchronize()
        check(f"o[{t}]", o, oref, "bf16")
    check("S", S, Sr, "bf16")
    check("p", p, pr, "bf16")


@pytest.mark.parametrize("variant,pc", [("diag", True), ("iso", False), ("iso", True)])
@pytest.mark.parametrize("logits", [False, True])
def test_fused_backward_bf16_gradients_every_instantiation(kdn, variant, pc, logits):
    """bf16-stored gradients from every fused backward instantiation: both
    variants, one or per-channel isotropic decay, post-activation and logit
    gates, on a ragged T; each gradient meets the bf16 rule plus its own
    rounding."""
    from kdn_gpu_util import check_stored_bf16
    B, T, H = 1, 140, 2
    ins = make_inputs(variant, B, T, H, 128, 128, dtype="bf16", seed=97, s0_std=0.05,
                      p0_range=(0.5, 2.0), per_channel_decay=pc, with_grad=True)
    kw, okw = {}, {}
    if logits:
        ins = _logits(ins, "bf16", 101)
        kw = dict(gates=kdn.KDN_GATES_LOGITS, r_min=R_MIN)
        okw = dict(gates="logits", r_min=R_MIN)
    _, bwd, _, _ = _fns(kdn, variant)
    d = to_dev(ins)
    grads = bwd(*[d[n] for n in NAMES], d["S0"], d["p0"], d["dO"], out_dtype=torch.bfloat16, **kw)
    torch.cuda.synchronize()
    gref = oracle.bwd(variant, *[ins[n] for n in NAMES], ins["S0"], ins["p0"], ins["dO"], **okw)
    for n in ("dq", "dk", "dv", "dg", "domega", "dr"):
        assert grads[n].dtype == torch.bfloat16
        check_stored_bf16(n, grads[n], gref[n])
    for n in ("dS0", "dp0"):
        check(n, grads[n], gref[n], "bf16")
