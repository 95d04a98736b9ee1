"""The allocation-free Diagonal-KDN forward (kdn_diag_fwd_noalloc).

It exists for callers that are given only input and output buffers and may
not call cudaMalloc (a latency-critical thread where an allocation can stall
on a device synchronisation, or a framework that forbids allocations outside
its own allocator).  Its scratch is a fixed array inside the library, so this
test checks, through the C ABI, that consecutive calls (each reusing the array
the previous one left behind) give the same results as the regular workspace
entry point, within the float32 parity tolerance, and match the fp64 oracle
within the tolerance of their input dtype; that the status word kept in the
array is readable through kdn_noalloc_device_status; and that a problem too
large for the array is refused.

This file is collected last on purpose: if it fails, a run that stops at the
first failure has already run every other test.
"""
import ctypes

import pytest
import torch

import oracle
from kdn_inputs import make_inputs
from kdn_gpu_util import check, err_ratio, to_dev

pytestmark = pytest.mark.gpu

NAMES = ("q", "k", "v", "g", "omega", "r")
SCRATCH_BYTES = 32 << 20  # KDN_NOALLOC_SCRATCH_BYTES in include/kdn.h


@pytest.fixture(scope="module")
def kdn():
    from paper_2609_07816_gb300 import build
    build.build()
    import paper_2609_07816_gb300 as m
    torch.cuda.init()
    return m


def _noalloc(kdn, d, o, ST, pT):
    desc = kdn.make_desc(*d["q"].shape[:3], d["q"].shape[3], d["v"].shape[3], d["q"].dtype)
    p = lambda t: None if t is None else ctypes.c_void_p(t.data_ptr())
    return kdn.lib().kdn_diag_fwd_noalloc(
        ctypes.byref(desc), *[p(d[n]) for n in NAMES], p(d["S0"]), p(d["p0"]), p(o), p(ST),
        p(pT), ctypes.c_void_p(torch.cuda.current_stream().cuda_stream))


def _check_against_workspace_call(kdn, shape, dtype):
    B, T, H, dk, dv, seed = shape
    ins = make_inputs("diag", B, T, H, dk, dv, dtype=dtype, seed=seed, s0_std=0.05,
                      p0_range=(0.5, 2.0))
    d = to_dev(ins)
    desc = kdn.make_desc(B, T, H, dk, dv, d["q"].dtype)
    assert kdn.workspace_bytes(desc, 0) <= SCRATCH_BYTES
    o_ref, ST_ref, pT_ref = kdn.kdn_diag_fwd(*[d[n] for n in NAMES], d["S0"], d["p0"])
    o = torch.full_like(o_ref, float("nan"))
    ST = torch.full_like(ST_ref, float("nan"))
    pT = torch.full_like(pT_ref, float("nan"))
    assert _noalloc(kdn, d, o, ST, pT) == kdn.KDN_OK
    assert kdn.kdn_noalloc_device_status() == kdn.KDN_OK
    torch.cuda.synchronize()
    for got, ref in ((o, o_ref), (ST, ST_ref), (pT, pT_ref)):
        assert err_ratio(got, ref.double().cpu().numpy()) <= 1e-4
    exact = oracle.fwd("diag", *[ins[n] for n in NAMES], ins["S0"], ins["p0"])
    for name, got in (("o", o), ("ST", ST), ("pT", pT)):
        check(name, got, exact[name], dtype)


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_noalloc_matches_workspace_entry_point_twice(kdn, dtype):
    # two different problems, then (bf16) one served by the sequence-parallel forward
    shapes = [(2, 150, 2, 128, 128, 3), (1, 97, 3, 64, 32, 4), (1, 2048, 2, 128, 128, 5)]
    for shape in shapes:
        _check_against_workspace_call(kdn, shape, dtype)


def test_noalloc_same_problem_twice_after_a_larger_one(kdn):
    """The array keeps whatever the previous call left: the same problem run
    twice in a row, the first time right after a larger problem filled more of
    the array, gives the workspace entry point's results both times."""
    _check_against_workspace_call(kdn, (1, 4096, 2, 128, 128, 6), "bf16")
    _check_against_workspace_call(kdn, (1, 2048, 2, 128, 128, 5), "bf16")
    _check_against_workspace_call(kdn, (1, 2048, 2, 128, 128, 5), "bf16")


def test_noalloc_status_word_is_readable(kdn):
    """A chunk whose cumulative decay leaves a fused kernel's range is reported
    in the status word kept in the library's array, through
    kdn_noalloc_device_status, which then clears it.  The problem (B=1, H=2,
    T=2048) is served by the sequence-parallel forward, whose segment passes
    take exp(G_C) >= 1e-36; alpha = e^-3 gives exp(G_C) = e^-192."""
    ins = make_inputs("diag", 1, 2048, 2, 128, 128, dtype="bf16", seed=3)
    ins["g"][...] = -3.0
    d = to_dev(ins)
    o = torch.empty(1, 2048, 2, 128, dtype=torch.float32, device="cuda")
    assert _noalloc(kdn, d, o, None, None) == kdn.KDN_OK
    assert kdn.kdn_noalloc_device_status() == kdn.KDN_ERR_RANGE
    assert kdn.kdn_noalloc_device_status() == kdn.KDN_OK


def test_noalloc_rejects_problems_larger_than_its_scratch(kdn):
    B, T, H = 4, 8192, 8   # float32 activations take the workspace-heavy chunked path
    desc = kdn.make_desc(B, T, H, 128, 128, torch.float32)
    assert kdn.workspace_bytes(desc, 0) > SCRATCH_BYTES
    fake = ctypes.c_void_p(1 << 20)  # never dereferenced: the call must refuse first
    st = kdn.lib().kdn_diag_fwd_noalloc(ctypes.byref(desc), *([fake] * 11), None)
    assert st == kdn.KDN_ERR_WORKSPACE
