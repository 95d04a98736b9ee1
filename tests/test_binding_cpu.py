"""The Python binding's argument checks, on the CPU.

Every tensor the binding hands to the C ABI becomes a raw device pointer, so
the binding refuses, before any launch, a tensor that is not on a CUDA device,
not contiguous, of another dtype than the library reads or writes there, or of
another element count than the descriptor implies.  These tests drive every
entry point with fake CUDA tensors (shapes and dtypes only, no device) and a
stand-in for the library that records its calls: the call patterns of the GPU
tests and the benchmark must reach the library, and each kind of bad argument
must be refused without reaching it.
"""
import contextlib

import pytest
import torch

fake_tensor = pytest.importorskip("torch._subclasses.fake_tensor")

import paper_2609_07816_gb300 as kdn  # noqa: E402

BF, F32 = torch.bfloat16, torch.float32


class FakeLib:
    """Accepts every entry point and records its name; sizes come back as 4096 bytes."""

    def __init__(self):
        self.calls = []

    def __getattr__(self, name):
        if name.endswith("_bytes"):
            return lambda *a: 4096
        if name == "kdn_status_string":
            return lambda s: b"fake"

        def call(*args):
            self.calls.append(name)
            return kdn.KDN_OK
        return call


@pytest.fixture
def fake(monkeypatch):
    lib = FakeLib()
    monkeypatch.setattr(kdn, "lib", lambda: lib)
    monkeypatch.setattr(kdn, "_ptr", lambda t: None)
    monkeypatch.setattr(kdn, "_stream", lambda s: None)
    with fake_tensor.FakeTensorMode(allow_non_fake_inputs=True):
        yield lib


def acts(variant, B, T, H, dk, dv, dtype=BF, per_channel=True, dev="cuda"):
    e = lambda *s: torch.empty(*s, dtype=dtype, device=dev)
    gshape = (B, T, H, dk) if (variant == "diag" or per_channel) else (B, T, H)
    wshape = (B, T, H, dk) if variant == "diag" else (B, T, H)
    return [e(B, T, H, dk), e(B, T, H, dk), e(B, T, H, dv), e(*gshape), e(*wshape), e(B, T, H)]


def state(variant, B, H, dk, dv):
    S = torch.empty(B, H, dk, dv, dtype=F32, device="cuda")
    p = torch.empty((B, H, dk) if variant == "diag" else (B, H), dtype=F32, device="cuda")
    return S, p


FNS = {"diag": (kdn.kdn_diag_fwd, kdn.kdn_diag_bwd, kdn.kdn_diag_fwd_save,
                kdn.kdn_diag_bwd_saved, kdn.kdn_diag_beta_eff, kdn.kdn_diag_decode_step),
       "iso": (kdn.kdn_iso_fwd, kdn.kdn_iso_bwd, kdn.kdn_iso_fwd_save,
               kdn.kdn_iso_bwd_saved, kdn.kdn_iso_beta_eff, kdn.kdn_iso_decode_step)}


@pytest.mark.parametrize("variant,pc", [("diag", True), ("iso", False), ("iso", True)])
def test_call_patterns_of_the_tests_and_bench_reach_the_library(fake, variant, pc):
    fwd, bwd, fsave, bsaved, beff, dec = FNS[variant]
    B, T, H, d = 2, 150, 3, 128
    x = acts(variant, B, T, H, d, d, per_channel=pc)
    S0, p0 = state(variant, B, H, d, d)
    dO = torch.empty(B, T, H, d, dtype=BF, device="cuda")
    fwd(*x)
    fwd(*x, S0, p0, chunk=32, want_state=False)
    fwd(*x, S0, p0, out_dtype=BF, gates=kdn.KDN_GATES_LOGITS, r_min=0.01)
    ws = torch.empty(256, dtype=torch.uint8, device="cuda")
    o = torch.empty(B, T, H, d, dtype=BF, device="cuda")
    fwd(*x, o=o, ST=S0.clone(), pT=p0.clone(), workspace=ws, out_dtype=BF)
    f32 = acts(variant, 1, 75, 2, 32, 32, dtype=F32, per_channel=pc)
    fwd(*f32, *state(variant, 1, 2, 32, 32))
    empty = [t[:, :0].contiguous() for t in x]
    fwd(*empty, S0, p0)
    fwd(*empty)
    bwd(*x, S0, p0, dO)
    bwd(*x, S0, p0, dO, *state(variant, B, H, d, d), out_dtype=BF)
    bwd(*f32, None, None, torch.empty(1, 75, 2, 32, dtype=F32, device="cuda"))
    _, _, _, saved = fsave(*x, S0, p0)
    grads = {n: torch.empty(t.shape, dtype=BF, device="cuda")
             for n, t in zip(("dq", "dk", "dv", "dg", "domega", "dr"), x)}
    fsave(*x, o=o, want_state=False, saved=saved, workspace=ws, out_dtype=BF)
    bsaved(*x, saved, dO, grads=grads, want_state_grads=False, workspace=ws, out_dtype=BF)
    bsaved(*x, saved, dO, *state(variant, B, H, d, d))
    beff(x[1], x[2], x[3], x[5], saved)
    # decode: per-step inputs without T, slices of stacked steps, o written in place
    steps = 4
    xs = [torch.empty(steps, *t[:, 0].shape, dtype=BF, device="cuda") for t in x]
    S, p = state(variant, B, H, d, d)
    od = torch.empty(steps, B, H, d, dtype=F32, device="cuda")
    for i in range(steps):
        dec(*[t[i] for t in xs], S, p, o=od[i])
    dec(*[t[0] for t in xs], S, p)
    if variant == "diag":
        kdn.kdn_diag_fwd_noalloc(*x, S0, p0, o=torch.empty(B, T, H, d, dtype=F32, device="cuda"))
    kdn.kdn_get_device_status(ws)
    kdn.kdn_selftest_wait_timeout(ws)
    assert len(fake.calls) >= 18


def _refused(fake, fn, *args, exc=(ValueError, TypeError), **kw):
    n = len(fake.calls)
    with pytest.raises(exc):
        fn(*args, **kw)
    assert len(fake.calls) == n, "a refused call must not reach the library"


def test_bad_tensors_are_refused_before_the_library(fake):
    B, T, H, d = 1, 64, 2, 128
    x = acts("diag", B, T, H, d, d)
    S0, p0 = state("diag", B, H, d, d)
    dO = torch.empty(B, T, H, d, dtype=BF, device="cuda")

    def with_(i, t):
        y = list(x)
        y[i] = t
        return y

    host = torch.empty(B, T, H, d, dtype=BF, device="cpu")
    _refused(fake, kdn.kdn_diag_fwd, *with_(0, host), exc=ValueError)          # host memory
    _refused(fake, kdn.kdn_diag_fwd, *with_(1, x[1].transpose(1, 2)), exc=ValueError)  # strided
    _refused(fake, kdn.kdn_diag_fwd, *with_(2, x[2].float()), exc=TypeError)   # mixed dtypes
    _refused(fake, kdn.kdn_diag_fwd, *with_(4, x[4][..., :64].contiguous()), exc=ValueError)
    _refused(fake, kdn.kdn_diag_fwd, *x, S0.double(), p0, exc=TypeError)
    _refused(fake, kdn.kdn_diag_fwd, *x, S0[:, :, :64].contiguous(), p0, exc=ValueError)
    _refused(fake, kdn.kdn_diag_fwd, *x, o=torch.empty(B, T, H, d, dtype=BF, device="cuda"),
             exc=TypeError)                                                     # o vs out_dtype
    _refused(fake, kdn.kdn_diag_fwd, *x, o=torch.empty(B, T, H, 64, device="cuda"),
             exc=ValueError)                                                    # o too small
    _refused(fake, kdn.kdn_diag_fwd, *x,
             workspace=torch.empty(64, dtype=F32, device="cuda"), exc=TypeError)
    _refused(fake, kdn.kdn_diag_bwd, *x, S0, p0, dO[:, :32].contiguous(), exc=ValueError)
    grads = {n: torch.empty(t.shape, dtype=F32, device="cuda")
             for n, t in zip(("dq", "dk", "dv", "dg", "domega", "dr"), x)}
    grads["dq"] = torch.empty(B, T, H, 64, dtype=F32, device="cuda")
    _refused(fake, kdn.kdn_diag_bwd, *x, S0, p0, dO, grads=grads, exc=ValueError)
    _refused(fake, kdn.kdn_diag_bwd_saved, *x, torch.empty(256, dtype=F32, device="cuda"), dO,
             exc=TypeError)                                                     # saved as bytes
    _refused(fake, kdn.kdn_diag_fwd_noalloc, *x, o=host.float(), exc=ValueError)
    xs = [t[:, 0].contiguous() for t in x]
    _refused(fake, kdn.kdn_diag_decode_step, *xs, S0.double(), p0, exc=TypeError)
    _refused(fake, kdn.kdn_diag_decode_step, *xs, S0, p0.cpu(), exc=ValueError)
    _refused(fake, kdn.kdn_get_device_status, torch.empty(256, dtype=torch.uint8), exc=ValueError)
    assert fake.calls == []
