"""C ABI checks that need no GPU: the library builds and loads, exports every
entry point that include/kdn.h declares, sizes workspaces, and rejects bad
arguments before any CUDA call is made."""
import ctypes
import math
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def kdn():
    from paper_2609_07816_gb300 import build
    build.build()
    import paper_2609_07816_gb300 as m
    return m


def _header_functions():
    text = open(os.path.join(ROOT, "include", "kdn.h")).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(kdn_[a-z_0-9]+)\s*\(", text)))


def test_exports_every_declared_symbol(kdn):
    names = _header_functions()
    assert len(names) >= 11
    L = ctypes.CDLL(kdn.LIB_PATH)
    for n in names:
        assert hasattr(L, n), n
    assert set(names) == set(kdn.EXPORTED)


def test_version_and_status_strings(kdn):
    assert kdn.lib().kdn_version() >= 100
    for code, name in enumerate(["KDN_OK", "KDN_ERR_INVALID_ARG", "KDN_ERR_UNSUPPORTED",
                                 "KDN_ERR_WORKSPACE", "KDN_ERR_CUDA", "KDN_ERR_TIMEOUT",
                                 "KDN_ERR_RANGE"]):
        assert kdn.status_string(code) == name
    assert kdn.status_string(99) == "KDN_ERR_UNKNOWN"


def test_workspace_sizes(kdn):
    d = kdn.make_desc(2, 100, 3, 64, 32, kdn.KDN_BF16)
    f0, b0 = kdn.workspace_bytes(d, 0), kdn.workspace_bytes(d, 0, True)
    f1 = kdn.workspace_bytes(d, 1)
    assert 0 < f0 < b0 and f1 > 0
    assert f0 % 256 == 0 and b0 % 256 == 0
    bad = kdn.make_desc(2, 100, 3, 96, 32, kdn.KDN_BF16)
    assert kdn.workspace_bytes(bad, 0) == 0
    # workspace grows linearly in T (per-chunk intermediates)
    d2 = kdn.make_desc(2, 200, 3, 64, 32, kdn.KDN_BF16)
    assert kdn.workspace_bytes(d2, 0) > f0


FAKE = ctypes.c_void_p(1 << 20)          # 16-byte aligned, never dereferenced
MIS = ctypes.c_void_p((1 << 20) + 4)     # misaligned


def _fwd(kdn, desc, ptrs=None, ws=FAKE, ws_bytes=1 << 40):
    p = ptrs or [FAKE] * 11
    return kdn.lib().kdn_diag_fwd(ctypes.byref(desc), *p, ws, ws_bytes, None)


def test_rejects_bad_descriptors_before_launch(kdn):
    L = kdn.lib()
    assert L.kdn_diag_fwd(None, *([FAKE] * 11), FAKE, 1 << 40, None) == kdn.KDN_ERR_INVALID_ARG
    cases = [
        (dict(dk=96), kdn.KDN_ERR_UNSUPPORTED),
        (dict(dv=48), kdn.KDN_ERR_UNSUPPORTED),
        (dict(dk=0), kdn.KDN_ERR_INVALID_ARG),
        (dict(T=-1), kdn.KDN_ERR_INVALID_ARG),
        (dict(B=-2), kdn.KDN_ERR_INVALID_ARG),
        (dict(chunk=48), kdn.KDN_ERR_INVALID_ARG),
        (dict(dtype=7), kdn.KDN_ERR_INVALID_ARG),
        (dict(out_dtype=3), kdn.KDN_ERR_INVALID_ARG),
        (dict(mu=math.nan), kdn.KDN_ERR_INVALID_ARG),
        (dict(scale=math.inf), kdn.KDN_ERR_INVALID_ARG),
        (dict(gates=2), kdn.KDN_ERR_INVALID_ARG),
        (dict(gates=-1), kdn.KDN_ERR_INVALID_ARG),
        (dict(gates=kdn.KDN_GATES_LOGITS, r_min=-0.01), kdn.KDN_ERR_INVALID_ARG),
        (dict(gates=kdn.KDN_GATES_LOGITS, r_min=math.inf), kdn.KDN_ERR_INVALID_ARG),
        (dict(gates=kdn.KDN_GATES_LOGITS, r_min=math.nan), kdn.KDN_ERR_INVALID_ARG),
    ]
    for over, want in cases:
        kw = dict(B=1, T=10, H=1, dk=32, dv=32, dtype=kdn.KDN_F32)
        kw.update(over)
        d = kdn.make_desc(kw["B"], kw["T"], kw["H"], kw["dk"], kw["dv"], kw["dtype"],
                          chunk=kw.get("chunk", 0), mu=kw.get("mu"), scale=kw.get("scale"),
                          out_dtype=kw.get("out_dtype", 0), gates=kw.get("gates", 0),
                          r_min=kw.get("r_min", 0.01))
        assert _fwd(kdn, d) == want, over
    # r_min is not read with post-activation gates
    d = kdn.make_desc(1, 10, 1, 32, 32, kdn.KDN_F32, r_min=math.nan)
    assert kdn.workspace_bytes(d, 0) > 0


def test_size_limits(kdn):
    """The largest problems a call takes (T = 2^21, B*T*H = 2^31 - 1 token-heads)
    get a workspace size; one token or sequence more is refused as unsupported,
    before any CUDA call.  No call here launches anything."""
    ok = [(1, 1 << 21, 1), (1023, 1 << 21, 1), (2, 1 << 20, 1023)]
    over = [(1, (1 << 21) + 1, 1), (1024, 1 << 21, 1), (1 << 16, 1, 1 << 10)]
    for B, T, H in ok:
        assert B * T * H <= (1 << 31) - 1
        assert kdn.workspace_bytes(kdn.make_desc(B, T, H, 32, 32, kdn.KDN_F32), 0) > 0
    for B, T, H in over:
        d = kdn.make_desc(B, T, H, 32, 32, kdn.KDN_F32)
        assert kdn.workspace_bytes(d, 0) == 0
        assert _fwd(kdn, d) == kdn.KDN_ERR_UNSUPPORTED


def test_rejects_null_and_misaligned_pointers(kdn):
    d = kdn.make_desc(1, 10, 1, 32, 32, kdn.KDN_F32)
    for i in range(7):  # q, k, v, g, omega, r are required; S0, p0 optional; o required
        idx = i if i < 6 else 8
        p = [FAKE] * 11
        p[idx] = None
        assert _fwd(kdn, d, p) == kdn.KDN_ERR_INVALID_ARG, idx
        p[idx] = MIS
        assert _fwd(kdn, d, p) == kdn.KDN_ERR_INVALID_ARG, idx
    p = [FAKE] * 11
    p[6] = MIS  # optional S0 must still be aligned
    assert _fwd(kdn, d, p) == kdn.KDN_ERR_INVALID_ARG


def test_rejects_small_or_misaligned_workspace(kdn):
    d = kdn.make_desc(1, 10, 1, 32, 32, kdn.KDN_F32)
    need = kdn.workspace_bytes(d, 0)
    assert _fwd(kdn, d, ws_bytes=need - 1) == kdn.KDN_ERR_WORKSPACE
    assert _fwd(kdn, d, ws=None, ws_bytes=need) == kdn.KDN_ERR_WORKSPACE
    assert _fwd(kdn, d, ws=ctypes.c_void_p((1 << 20) + 16), ws_bytes=need) == \
        kdn.KDN_ERR_WORKSPACE


def test_backward_and_decode_validate(kdn):
    L = kdn.lib()
    d = kdn.make_desc(1, 10, 1, 32, 32, kdn.KDN_BF16)
    p = [FAKE] * 20
    p[15] = None  # domega is required
    assert L.kdn_iso_bwd(ctypes.byref(d), *p, FAKE, 1 << 40, None) == kdn.KDN_ERR_INVALID_ARG
    p = [FAKE] * 20
    p[19] = MIS  # dmu is optional but must be aligned
    assert L.kdn_iso_bwd(ctypes.byref(d), *p, FAKE, 1 << 40, None) == kdn.KDN_ERR_INVALID_ARG
    q = [FAKE] * 9
    q[7] = None  # p (state) is required
    assert L.kdn_diag_decode_step(ctypes.byref(d), *q, None) == kdn.KDN_ERR_INVALID_ARG
    bad = kdn.make_desc(1, 1, 1, 32, 40, kdn.KDN_BF16)
    assert L.kdn_iso_decode_step(ctypes.byref(bad), *([FAKE] * 9), None) == \
        kdn.KDN_ERR_UNSUPPORTED
    iso = kdn.make_desc(1, 10, 1, 32, 32, kdn.KDN_BF16, decay_per_channel=3)
    assert L.kdn_iso_fwd(ctypes.byref(iso), *([FAKE] * 11), FAKE, 1 << 40, None) == \
        kdn.KDN_ERR_INVALID_ARG


def test_product_package_does_not_import_oracle():
    pkg = os.path.join(ROOT, "paper_2609_07816_gb300")
    for dirpath, _, files in os.walk(pkg):
        for f in files:
            if f.endswith((".py", ".cu", ".cuh", ".h")):
                text = open(os.path.join(dirpath, f)).read()
                assert "oracle" not in text.lower().replace("oracle-free", ""), f


def test_kernel_launch_query(kdn):
    d = kdn.make_desc(2, 100, 3, 64, 32, kdn.KDN_BF16)
    f, b, dec = (kdn.kdn_kernel_launches(d, 0, op) for op in (0, 1, 2))
    assert f >= 1 and b > f and dec == 1
    assert kdn.kdn_kernel_launches(d, 1, 0) >= 1
    assert kdn.kdn_kernel_launches(d, 0, 7) == -1
    assert kdn.kdn_kernel_launches(kdn.make_desc(1, 4, 1, 96, 32, 0), 0, 0) == -1


def test_fused_path_launches_and_workspace(kdn):
    """bf16, dk = dv = 128: the fused forward is one launch; the fused backward
    (both variants) is two (context-saving forward + reverse sweep) and its
    workspace holds a 162 KB context record per chunk (S_in, R, -W, A_qk, A and
    Y as 16-bit tiles, phat and gamma in fp32, per-token scalars) and 128 floats
    of uncertainty per chunk."""
    B, T, H = 2, 130, 3
    d = kdn.make_desc(B, T, H, 128, 128, kdn.KDN_BF16)
    assert kdn.kdn_kernel_launches(d, 0, 0) == 1
    assert kdn.kdn_kernel_launches(d, 0, 1) == 2
    NC = (T + 63) // 64
    need = 256 + B * H * NC * 165888 + B * H * NC * 128 * 4
    assert kdn.workspace_bytes(d, 0, True) == need
    # the isotropic backward is fused too; the 32-token chunk keeps the general kernels
    assert kdn.kdn_kernel_launches(d, 1, 1) == 2
    assert kdn.workspace_bytes(d, 1, True) == need
    d32 = kdn.make_desc(B, T, H, 128, 128, kdn.KDN_BF16, chunk=32)
    assert kdn.kdn_kernel_launches(d32, 0, 1) > 2


def _seg_bytes(B, T, H, P, variant):
    r = lambda x: (x + 255) // 256 * 256
    Pn = 128 if variant == 0 else 1
    BH, NC = B * H, T // 64
    # summaries, 2 uncertainty buffers, the exit memories Sv and Phi, the fp16
    # images of the entry memories and the fp16 output of the transition pass
    # (o is float32 here, so it holds o_v)
    return (r(BH * NC * Pn * 16) + 2 * r(BH * P * Pn * 4) + 2 * r(BH * P * 128 * 128 * 4)
            + r(BH * P * 32768) + r(B * T * H * 128 * 2))


@pytest.mark.parametrize("B,T,H,P", [
    (1, 65536, 16, 8),    # long context: 1024 chunks cut into 8 segments of 128
    (1, 2048, 2, 4),      # 32 chunks: 4 segments of 8
    (2, 2560, 1, 5),      # 40 chunks: 5 segments of 8
    (1, 2304, 2, 4),      # 36 chunks: 4 segments of 9
    (2, 4096, 1, 8),
    (8, 4096, 16, 1),     # B*H = 128: already one CTA per SM, no segments
    (1, 2047, 2, 1),      # T not a multiple of 64
    (1, 1536, 2, 1),      # 24 chunks: too short for 4 segments of 8
])
def test_sequence_parallel_forward_selection(kdn, B, T, H, P):
    """The plain bf16 d = 128 forward of few long sequences is cut into P
    segments (the largest divisor of the chunk count with B*H*P <= 152 and
    segments of at least 8 chunks, P >= 4): five launches and the segment
    buffers after the status word; otherwise one fused launch."""
    for variant in (0, 1):
        d = kdn.make_desc(B, T, H, 128, 128, kdn.KDN_BF16)
        if P > 1:
            assert kdn.kdn_kernel_launches(d, variant, 0) == 5
            assert kdn.workspace_bytes(d, variant) == 256 + _seg_bytes(B, T, H, P, variant)
        else:
            assert kdn.kdn_kernel_launches(d, variant, 0) == 1
            assert kdn.workspace_bytes(d, variant) == 256
        # the 32-token chunk keeps the general kernels
        d32 = kdn.make_desc(B, T, H, 128, 128, kdn.KDN_BF16, chunk=32)
        assert kdn.kdn_kernel_launches(d32, variant, 0) not in (1, 5)


def test_training_pair_validation(kdn):
    """kdn_diag_fwd_save / kdn_diag_bwd_saved: served only for the fused shapes;
    the saved buffer is checked for size and alignment before anything runs."""
    L = kdn.lib()
    B, T, H = 2, 130, 3
    d = kdn.make_desc(B, T, H, 128, 128, kdn.KDN_BF16)
    n = kdn.saved_bytes(d)
    assert n == B * H * 3 * (165888 + 512)
    assert kdn.saved_bytes(d, 1) == n
    assert kdn.saved_bytes(kdn.make_desc(B, T, H, 64, 128, kdn.KDN_BF16)) == 0
    assert kdn.saved_bytes(kdn.make_desc(B, T, H, 128, 128, kdn.KDN_F32)) == 0
    assert kdn.kdn_kernel_launches(d, 0, 3) == 1 and kdn.kdn_kernel_launches(d, 0, 4) == 1
    assert kdn.kdn_kernel_launches(d, 1, 3) == 1 and kdn.kdn_kernel_launches(d, 1, 4) == 1
    assert kdn.kdn_kernel_launches(kdn.make_desc(B, T, H, 64, 128, kdn.KDN_BF16), 1, 3) == -1

    def fwd_save(desc, saved=FAKE, saved_bytes=1 << 40):
        return L.kdn_diag_fwd_save(ctypes.byref(desc), *([FAKE] * 11), saved, saved_bytes, FAKE,
                                   1 << 40, None)

    def bwd_saved(desc, saved=FAKE, saved_bytes=1 << 40):
        return L.kdn_diag_bwd_saved(ctypes.byref(desc), *([FAKE] * 6), saved, saved_bytes,
                                    *([FAKE] * 12), FAKE, 1 << 40, None)

    for fn in (fwd_save, bwd_saved):
        assert fn(kdn.make_desc(B, T, H, 64, 128, kdn.KDN_BF16)) == kdn.KDN_ERR_UNSUPPORTED
        assert fn(d, saved_bytes=n - 1) == kdn.KDN_ERR_WORKSPACE
        assert fn(d, saved=MIS) in (kdn.KDN_ERR_INVALID_ARG, kdn.KDN_ERR_WORKSPACE)
        assert fn(d, saved=None) == kdn.KDN_ERR_INVALID_ARG


def test_beta_eff_validation(kdn):
    """kdn_*_beta_eff reads a saved training context: served for the same
    descriptors as the training pair, pointers and the saved size are checked
    before anything runs, T = 0 is a no-op (no GPU needed for any of this)."""
    L = kdn.lib()
    B, T, H = 2, 130, 3
    d = kdn.make_desc(B, T, H, 128, 128, kdn.KDN_BF16)
    n = kdn.saved_bytes(d)
    assert kdn.kdn_kernel_launches(d, 0, 5) == 1 and kdn.kdn_kernel_launches(d, 1, 5) == 1
    assert kdn.kdn_kernel_launches(kdn.make_desc(B, T, H, 128, 128, kdn.KDN_F32), 0, 5) == -1
    for fn in (L.kdn_diag_beta_eff, L.kdn_iso_beta_eff):
        def call(desc, saved=FAKE, saved_bytes=1 << 40, r=FAKE, out=FAKE):
            return fn(ctypes.byref(desc), saved, saved_bytes, r, out, None)
        assert call(kdn.make_desc(B, T, H, 64, 128, kdn.KDN_BF16)) == kdn.KDN_ERR_UNSUPPORTED
        assert call(kdn.make_desc(B, T, H, 128, 128, kdn.KDN_F32)) == kdn.KDN_ERR_UNSUPPORTED
        assert call(d, saved=None) == kdn.KDN_ERR_INVALID_ARG
        assert call(d, r=None) == kdn.KDN_ERR_INVALID_ARG
        assert call(d, out=MIS) == kdn.KDN_ERR_INVALID_ARG
        assert call(d, saved_bytes=n - 1) == kdn.KDN_ERR_WORKSPACE
        assert call(kdn.make_desc(B, 0, H, 128, 128, kdn.KDN_BF16), saved=None) == kdn.KDN_OK
        assert call(d, saved=MIS) == kdn.KDN_ERR_INVALID_ARG


def test_wait_timeout_selftest_validates(kdn):
    """The device self-test of the bounded waits rejects a null or misaligned
    workspace before anything runs (no GPU needed)."""
    L = kdn.lib()
    assert L.kdn_selftest_wait_timeout(None, None) == kdn.KDN_ERR_INVALID_ARG
    assert L.kdn_selftest_wait_timeout(MIS, None) == kdn.KDN_ERR_INVALID_ARG
