"""GPU parity at the measured workload sizes, in the launch configuration the
benchmark uses (bf16 activations, float32 outputs, default chunk).  The GPU
computes every (batch, head); the oracle recomputes a sample of them one by
one, and the sampled outputs are compared element by element under
max|err| <= 2e-2 * RMS(oracle)."""
import numpy as np
import pytest
import torch

import oracle
from kdn_inputs import make_decode_inputs, make_inputs
from kdn_gpu_util import check, head_slice, to_dev

pytestmark = pytest.mark.gpu
NAMES = ("q", "k", "v", "g", "omega", "r")


@pytest.fixture(scope="module")
def kdn():
    from paper_2609_07816_gb300 import build
    build.build()
    import paper_2609_07816_gb300 as m
    torch.cuda.init()
    return m


def _sampled_fwd_check(kdn, variant, ins, heads):
    d = to_dev(ins)
    fwd = kdn.kdn_diag_fwd if variant == "diag" else kdn.kdn_iso_fwd
    o, ST, pT = fwd(*[d[n] for n in NAMES], d["S0"], d["p0"])
    torch.cuda.synchronize()
    for b, h in heads:
        sl = head_slice(ins, b, h)
        ref = oracle.fwd(variant, *[sl[n] for n in NAMES], sl["S0"], sl["p0"])
        check(f"o[{b},{h}]", o[b:b + 1, :, h:h + 1], ref["o"], "bf16")
        check(f"ST[{b},{h}]", ST[b:b + 1, h:h + 1], ref["ST"], "bf16")
        check(f"pT[{b},{h}]", pT[b:b + 1, h:h + 1], ref["pT"], "bf16")


def test_iso_750m_layer_shape(kdn):
    """Isotropic KDN, B=8 H=12 T=2048 d=128, scalar decay and noise."""
    ins = make_inputs("iso", 8, 2048, 12, 128, 128, dtype="bf16", seed=0,
                      per_channel_decay=False)
    _sampled_fwd_check(kdn, "iso", ins, [(0, 0), (3, 7), (7, 11)])


def test_iso_750m_layer_shape_backward(kdn):
    """Isotropic KDN backward, B=8 H=12 T=2048 d=128, scalar decay, dO ~ N(0,1)."""
    ins = make_inputs("iso", 8, 2048, 12, 128, 128, dtype="bf16", seed=0,
                      per_channel_decay=False, with_grad=True)
    d = to_dev(ins)
    gr = kdn.kdn_iso_bwd(*[d[n] for n in NAMES], None, None, d["dO"])
    torch.cuda.synchronize()
    for b, h in [(0, 0), (7, 11)]:
        sl = head_slice(ins, b, h)
        ref = oracle.bwd("iso", *[sl[n] for n in NAMES], None, None, sl["dO"])
        for n in ("dq", "dk", "dv", "dg", "domega", "dr"):
            check(f"{n}[{b},{h}]", gr[n][b:b + 1, :, h:h + 1], ref[n], "bf16")
        check(f"dS0[{b},{h}]", gr["dS0"][b:b + 1, h:h + 1], ref["dS0"], "bf16")
        check(f"dp0[{b},{h}]", gr["dp0"][b:b + 1, h:h + 1], ref["dp0"], "bf16")


def test_diag_1p3b_layer_shape_forward(kdn):
    """Diagonal KDN forward, B=8 H=16 T=4096 d=128."""
    ins = make_inputs("diag", 8, 4096, 16, 128, 128, dtype="bf16", seed=0)
    _sampled_fwd_check(kdn, "diag", ins, [(0, 0), (5, 9), (7, 15)])


def test_diag_1p3b_layer_shape_backward(kdn):
    """Diagonal KDN backward, B=8 H=16 T=4096 d=128, dO ~ N(0,1), no state cotangent."""
    ins = make_inputs("diag", 8, 4096, 16, 128, 128, dtype="bf16", seed=0, with_grad=True)
    d = to_dev(ins)
    gr = kdn.kdn_diag_bwd(*[d[n] for n in NAMES], None, None, d["dO"])
    torch.cuda.synchronize()
    for b, h in [(0, 0), (6, 13)]:
        sl = head_slice(ins, b, h)
        ref = oracle.bwd("diag", *[sl[n] for n in NAMES], None, None, sl["dO"])
        for n in ("dq", "dk", "dv", "dg", "domega", "dr"):
            x = gr[n][b:b + 1, :, h:h + 1]
            check(f"{n}[{b},{h}]", x, ref[n], "bf16")
        check(f"dS0[{b},{h}]", gr["dS0"][b:b + 1, h:h + 1], ref["dS0"], "bf16")
        check(f"dp0[{b},{h}]", gr["dp0"][b:b + 1, h:h + 1], ref["dp0"], "bf16")


@pytest.mark.parametrize("variant", ["diag", "iso"])
def test_long_context_shape(kdn, variant):
    """B=1 H=16 T=65536 d=128, S_0 ~ N(0, 0.02^2), p_0 ~ U(0.5, 2)."""
    ins = make_inputs(variant, 1, 65536, 16, 128, 128, dtype="bf16", seed=0, s0_std=0.02,
                      p0_range=(0.5, 2.0))
    _sampled_fwd_check(kdn, variant, ins, [(0, 4)])


@pytest.mark.parametrize("variant", ["diag", "iso"])
def test_decode_batch_shape(kdn, variant):
    """B=256 H=16 d=128 decode with fp32 state ~ N(0,0.02^2) / U(0.1,2), 6 steps."""
    steps = 6
    ins = make_decode_inputs(variant, 256, 16, 128, 128, steps, dtype="bf16", seed=0)
    S = torch.tensor(ins["S"], dtype=torch.float32, device="cuda")
    p = torch.tensor(ins["p"], dtype=torch.float32, device="cuda")
    fn = kdn.kdn_diag_decode_step if variant == "diag" else kdn.kdn_iso_decode_step
    outs = []
    for s in range(steps):
        x = {n: torch.tensor(ins[n][s], dtype=torch.bfloat16, device="cuda") for n in NAMES}
        outs.append(fn(*[x[n] for n in NAMES], S, p).clone())
    torch.cuda.synchronize()
    for b, h in [(0, 0), (100, 5), (255, 15)]:
        Sr, pr = ins["S"][b:b + 1, h:h + 1], ins["p"][b:b + 1, h:h + 1]
        for s in range(steps):
            o_ref, Sr, pr = oracle.decode_step(
                variant, *[ins[n][s][b:b + 1, h:h + 1] for n in NAMES], Sr, pr)
            check(f"o[{s}][{b},{h}]", outs[s][b:b + 1, h:h + 1], o_ref, "bf16")
        check(f"S[{b},{h}]", S[b:b + 1, h:h + 1], Sr, "bf16")
        check(f"p[{b},{h}]", p[b:b + 1, h:h + 1], pr, "bf16")
