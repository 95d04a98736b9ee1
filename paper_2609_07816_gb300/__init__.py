"""GB300 (sm_103a) Kalman Delta Network token mixers.

Thin Python binding of ``libkdn.so`` (C ABI in ``include/kdn.h``).  The
functions below carry the C entry points' names and only marshal arguments:
they check that every tensor is what the C ABI reads through its pointer (a
contiguous CUDA tensor of the expected dtype and element count), allocate
outputs and the scratch workspace with PyTorch (device memory is PyTorch's job
here), pass raw pointers and the current CUDA stream, and raise on any non-OK
status.  Every step of the computation runs in the library's
CUDA kernels; there is no CPU or PyTorch fallback, and importing a function
whose library is missing raises.

Layouts follow the C ABI: q, k [B,T,H,dk]; v [B,T,H,dv]; r [B,T,H];
diag g, omega [B,T,H,dk]; iso omega [B,T,H], g [B,T,H,dk] or [B,T,H];
S0 [B,H,dk,dv] float32; p0 diag [B,H,dk], iso [B,H] float32.
"""
from __future__ import annotations

import ctypes
import math
import os
import threading

import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libkdn.so")

KDN_OK, KDN_ERR_INVALID_ARG, KDN_ERR_UNSUPPORTED, KDN_ERR_WORKSPACE, KDN_ERR_CUDA, \
    KDN_ERR_TIMEOUT, KDN_ERR_RANGE = range(7)
KDN_F32, KDN_BF16 = 0, 1
KDN_GATES_POST, KDN_GATES_LOGITS = 0, 1
R_MIN_DEFAULT = 0.01  # the layer's observation-noise floor

_DTYPES = {torch.float32: KDN_F32, torch.bfloat16: KDN_BF16}


class kdn_desc_t(ctypes.Structure):
    _fields_ = [("B", ctypes.c_int), ("T", ctypes.c_int), ("H", ctypes.c_int),
                ("dk", ctypes.c_int), ("dv", ctypes.c_int), ("chunk", ctypes.c_int),
                ("dtype", ctypes.c_int), ("mu", ctypes.c_float), ("scale", ctypes.c_float),
                ("decay_per_channel", ctypes.c_int), ("out_dtype", ctypes.c_int),
                ("gates", ctypes.c_int), ("r_min", ctypes.c_float)]


class KdnError(RuntimeError):
    def __init__(self, status: int, where: str):
        self.status = status
        super().__init__(f"{where}: {status_string(status)}")


_lib = None
_lock = threading.Lock()

_P = ctypes.c_void_p
_SIG = {
    "kdn_version": ([], ctypes.c_int),
    "kdn_status_string": ([ctypes.c_int], ctypes.c_char_p),
    "kdn_fwd_workspace_bytes": ([ctypes.POINTER(kdn_desc_t), ctypes.c_int], ctypes.c_size_t),
    "kdn_bwd_workspace_bytes": ([ctypes.POINTER(kdn_desc_t), ctypes.c_int], ctypes.c_size_t),
    "kdn_diag_fwd": ([ctypes.POINTER(kdn_desc_t)] + [_P] * 12 + [ctypes.c_size_t, _P], ctypes.c_int),
    "kdn_iso_fwd": ([ctypes.POINTER(kdn_desc_t)] + [_P] * 12 + [ctypes.c_size_t, _P], ctypes.c_int),
    "kdn_diag_bwd": ([ctypes.POINTER(kdn_desc_t)] + [_P] * 21 + [ctypes.c_size_t, _P], ctypes.c_int),
    "kdn_iso_bwd": ([ctypes.POINTER(kdn_desc_t)] + [_P] * 21 + [ctypes.c_size_t, _P], ctypes.c_int),
    "kdn_diag_decode_step": ([ctypes.POINTER(kdn_desc_t)] + [_P] * 10, ctypes.c_int),
    "kdn_iso_decode_step": ([ctypes.POINTER(kdn_desc_t)] + [_P] * 10, ctypes.c_int),
    "kdn_diag_fwd_noalloc": ([ctypes.POINTER(kdn_desc_t)] + [_P] * 12, ctypes.c_int),
    "kdn_saved_bytes": ([ctypes.POINTER(kdn_desc_t), ctypes.c_int], ctypes.c_size_t),
    "kdn_diag_fwd_save": ([ctypes.POINTER(kdn_desc_t)] + [_P] * 12 + [ctypes.c_size_t, _P,
                                                                   ctypes.c_size_t, _P], ctypes.c_int),
    "kdn_diag_bwd_saved": ([ctypes.POINTER(kdn_desc_t)] + [_P] * 7 + [ctypes.c_size_t] + [_P] * 13
                           + [ctypes.c_size_t, _P], ctypes.c_int),
    "kdn_iso_fwd_save": ([ctypes.POINTER(kdn_desc_t)] + [_P] * 12 + [ctypes.c_size_t, _P,
                                                                  ctypes.c_size_t, _P], ctypes.c_int),
    "kdn_iso_bwd_saved": ([ctypes.POINTER(kdn_desc_t)] + [_P] * 7 + [ctypes.c_size_t] + [_P] * 13
                          + [ctypes.c_size_t, _P], ctypes.c_int),
    "kdn_diag_beta_eff": ([ctypes.POINTER(kdn_desc_t), _P, ctypes.c_size_t, _P, _P, _P], ctypes.c_int),
    "kdn_iso_beta_eff": ([ctypes.POINTER(kdn_desc_t), _P, ctypes.c_size_t, _P, _P, _P], ctypes.c_int),
    "kdn_kernel_launches": ([ctypes.POINTER(kdn_desc_t), ctypes.c_int, ctypes.c_int], ctypes.c_int),
    "kdn_get_device_status": ([_P, _P], ctypes.c_int),
    "kdn_noalloc_device_status": ([_P], ctypes.c_int),
    "kdn_selftest_wait_timeout": ([_P, _P], ctypes.c_int),
}
EXPORTED = tuple(_SIG)


def lib():
    """The loaded ``libkdn.so`` (ctypes), built beforehand by ``build.build()``."""
    global _lib
    with _lock:
        if _lib is None:
            if not os.path.exists(LIB_PATH):
                raise RuntimeError(f"{LIB_PATH} is missing: run paper_2609_07816_gb300.build."
                                   "build() first (there is no fallback implementation)")
            L = ctypes.CDLL(LIB_PATH)
            for name, (args, res) in _SIG.items():
                fn = getattr(L, name)
                fn.argtypes = args
                fn.restype = res
            _lib = L
    return _lib


def status_string(status: int) -> str:
    return lib().kdn_status_string(int(status)).decode()


def _check(status: int, where: str):
    if status != KDN_OK:
        raise KdnError(status, where)


def _ptr(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream(stream):
    s = torch.cuda.current_stream() if stream is None else stream
    return ctypes.c_void_p(s.cuda_stream)


def _code(dtype):
    return _DTYPES[dtype] if isinstance(dtype, torch.dtype) else int(dtype)


_TORCH = {KDN_F32: torch.float32, KDN_BF16: torch.bfloat16}


def _torch_dtype(dtype):
    return dtype if isinstance(dtype, torch.dtype) else _TORCH[int(dtype)]


def _arg(t, name, dtype=None, numel=None, required=True):
    """A tensor handed to the C ABI as a raw pointer: it must be device memory (a
    CUDA tensor), dense in the ABI's row-major layout (contiguous), of the dtype
    the library reads or writes there and of the element count the descriptor
    implies.  Anything else would make the kernels read or write the wrong
    memory, so it is refused here, before any launch."""
    if t is None:
        if required:
            raise ValueError(f"{name} is required")
        return
    if not isinstance(t, torch.Tensor):
        raise TypeError(f"{name}: expected a torch.Tensor, got {type(t).__name__}")
    if not t.is_cuda:
        raise ValueError(f"{name}: must be a CUDA tensor (the kernels read device memory), "
                         f"got one on {t.device}")
    if not t.is_contiguous():
        raise ValueError(f"{name}: must be contiguous (the C ABI's row-major layout)")
    if dtype is not None and t.dtype != dtype:
        raise TypeError(f"{name}: dtype {t.dtype}, expected {dtype}")
    if numel is not None and t.numel() != numel:
        raise ValueError(f"{name}: {t.numel()} elements, expected {numel}")


def _check_inputs(variant, q, k, v, g, omega, r, dO=None, tokens=True):
    """The per-token inputs (and dO): one activation dtype, the ABI's layouts.
    ``tokens`` = False for the decode step, whose inputs drop the T axis."""
    _arg(q, "q")
    if q.dtype not in _DTYPES:
        raise TypeError(f"q: dtype {q.dtype}, expected torch.float32 or torch.bfloat16")
    if q.dim() != (4 if tokens else 3):
        raise ValueError(f"q: {q.dim()} dimensions, expected {4 if tokens else 3}")
    dk = q.shape[-1]
    n = q.numel() // dk if dk else 0
    _arg(v, "v", q.dtype)
    _arg(g, "g", q.dtype)
    dv = v.shape[-1]
    per_channel = variant == 0 or g.dim() == q.dim()
    for t, name, m in ((k, "k", dk), (v, "v", dv), (g, "g", dk if per_channel else 1),
                       (omega, "omega", dk if variant == 0 else 1), (r, "r", 1)):
        _arg(t, name, q.dtype, n * m)
    if dO is not None:
        _arg(dO, "dO", q.dtype, n * dv)


def _state_sizes(variant, q, v, tokens=True):
    B, H = q.shape[0], q.shape[2 if tokens else 1]
    dk, dv = q.shape[-1], v.shape[-1]
    return B * H * dk * dv, B * H * (dk if variant == 0 else 1)


def _check_grads(G, q, k, v, g, omega, r, out_dtype, ns, np_):
    """Gradient buffers: one per input, its element count, the output dtype;
    dS0, dp0 and dmu (optional) in float32."""
    od = _torch_dtype(out_dtype)
    for n, x in (("dq", q), ("dk", k), ("dv", v), ("dg", g), ("domega", omega), ("dr", r)):
        _arg(G.get(n), n, od, x.numel())
    _arg(G.get("dS0"), "dS0", torch.float32, ns, required=False)
    _arg(G.get("dp0"), "dp0", torch.float32, np_, required=False)
    _arg(G.get("dmu"), "dmu", torch.float32, q.shape[0] * q.shape[2], required=False)


def make_desc(B, T, H, dk, dv, dtype, *, chunk=0, mu=None, scale=None,
              decay_per_channel=1, out_dtype=KDN_F32, gates=KDN_GATES_POST,
              r_min=R_MIN_DEFAULT) -> kdn_desc_t:
    """``gates``: KDN_GATES_POST (g = log alpha, omega, r) or KDN_GATES_LOGITS
    (g, omega, r are the logits of sigmoid / softplus / r_min + softplus)."""
    return kdn_desc_t(B, T, H, dk, dv, chunk, _code(dtype), 0.0 if mu is None else float(mu),
                      math.nan if scale is None else float(scale), int(decay_per_channel),
                      _code(out_dtype), int(gates), float(r_min))


def _desc_from(variant, q, v, g, *, chunk, mu, scale, out_dtype, gates=KDN_GATES_POST,
               r_min=R_MIN_DEFAULT):
    B, T, H, dk = q.shape
    dv = v.shape[-1]
    pcd = 1 if variant == 0 else int(g.dim() == 4)
    return make_desc(B, T, H, dk, dv, q.dtype, chunk=chunk, mu=mu, scale=scale,
                     decay_per_channel=pcd, out_dtype=out_dtype,
        gates=gates, r_min=r_min)


def workspace_bytes(desc: kdn_desc_t, variant: int, backward: bool = False) -> int:
    fn = lib().kdn_bwd_workspace_bytes if backward else lib().kdn_fwd_workspace_bytes
    return int(fn(ctypes.byref(desc), int(variant)))


def alloc_workspace(desc, variant, backward=False, device=None):
    n = workspace_bytes(desc, variant, backward)
    return torch.empty(max(n, 256), dtype=torch.uint8, device=device or "cuda")


def _fwd(name, variant, q, k, v, g, omega, r, S0, p0, *, chunk, mu, scale, o, ST, pT,
         want_state, workspace, stream, out_dtype,
         gates=KDN_GATES_POST, r_min=R_MIN_DEFAULT):
    _check_inputs(variant, q, k, v, g, omega, r)
    desc = _desc_from(variant, q, v, g, chunk=chunk, mu=mu, scale=scale, out_dtype=out_dtype,
                      gates=gates, r_min=r_min)
    B, T, H, dk = q.shape
    dv = v.shape[-1]
    dev = q.device
    ns, np_ = _state_sizes(variant, q, v)
    _arg(S0, "S0", torch.float32, ns, required=False)
    _arg(p0, "p0", torch.float32, np_, required=False)
    if o is None:
        o = torch.empty(B, T, H, dv, dtype=out_dtype, device=dev)
    if want_state and ST is None:
        ST = torch.empty(B, H, dk, dv, dtype=torch.float32, device=dev)
    if want_state and pT is None:
        pT = torch.empty((B, H, dk) if variant == 0 else (B, H), dtype=torch.float32, device=dev)
    if workspace is None:
        workspace = alloc_workspace(desc, variant, False, dev)
    _arg(o, "o", _torch_dtype(out_dtype), B * T * H * dv)
    _arg(ST, "ST", torch.float32, ns, required=False)
    _arg(pT, "pT", torch.float32, np_, required=False)
    _arg(workspace, "workspace", torch.uint8)
    st = getattr(lib(), name)(ctypes.byref(desc), _ptr(q), _ptr(k), _ptr(v), _ptr(g),
                              _ptr(omega), _ptr(r), _ptr(S0), _ptr(p0), _ptr(o), _ptr(ST),
                              _ptr(pT), _ptr(workspace), workspace.numel(), _stream(stream))
    _check(st, name)
    return o, ST, pT


def kdn_diag_fwd(q, k, v, g, omega, r, S0=None, p0=None, *, chunk=0, mu=None, scale=None,
                 o=None, ST=None, pT=None, want_state=True, workspace=None, stream=None,
                 out_dtype=torch.float32, gates=KDN_GATES_POST,
                 r_min=R_MIN_DEFAULT):
    """Diagonal KDN forward (Prop. 3).  Returns (o, ST, pT)."""
    return _fwd("kdn_diag_fwd", 0, q, k, v, g, omega, r, S0, p0, chunk=chunk, mu=mu,
                scale=scale, o=o, ST=ST, pT=pT, want_state=want_state, workspace=workspace,
                stream=stream, out_dtype=out_dtype,
        gates=gates, r_min=r_min)


def kdn_iso_fwd(q, k, v, g, omega, r, S0=None, p0=None, *, chunk=0, mu=None, scale=None,
                o=None, ST=None, pT=None, want_state=True, workspace=None, stream=None,
                 out_dtype=torch.float32, gates=KDN_GATES_POST,
                 r_min=R_MIN_DEFAULT):
    """Isotropic KDN forward (Prop. 5).  g [B,T,H,dk] = per-channel decay, [B,T,H] = scalar."""
    return _fwd("kdn_iso_fwd", 1, q, k, v, g, omega, r, S0, p0, chunk=chunk, mu=mu,
                scale=scale, o=o, ST=ST, pT=pT, want_state=want_state, workspace=workspace,
                stream=stream, out_dtype=out_dtype,
        gates=gates, r_min=r_min)


def _bwd(name, variant, q, k, v, g, omega, r, S0, p0, dO, dST, dpT, *, chunk, mu, scale,
         grads, want_state_grads, workspace, stream, out_dtype,
         gates=KDN_GATES_POST, r_min=R_MIN_DEFAULT):
    _check_inputs(variant, q, k, v, g, omega, r, dO)
    desc = _desc_from(variant, q, v, g, chunk=chunk, mu=mu, scale=scale, out_dtype=out_dtype,
                      gates=gates, r_min=r_min)
    B, T, H, dk = q.shape
    dv = v.shape[-1]
    dev = q.device
    ns, np_ = _state_sizes(variant, q, v)
    for t, n, m in ((S0, "S0", ns), (p0, "p0", np_), (dST, "dST", ns), (dpT, "dpT", np_)):
        _arg(t, n, torch.float32, m, required=False)
    if grads is None:
        grads = {n: torch.empty(x.shape, dtype=out_dtype, device=dev) for n, x in
                 (("dq", q), ("dk", k), ("dv", v), ("dg", g), ("domega", omega), ("dr", r))}
        if want_state_grads:
            grads["dS0"] = torch.empty(B, H, dk, dv, dtype=torch.float32, device=dev)
            grads["dp0"] = torch.empty((B, H, dk) if variant == 0 else (B, H),
                                       dtype=torch.float32, device=dev)
            grads["dmu"] = torch.empty(B, H, dtype=torch.float32, device=dev)
    if workspace is None:
        workspace = alloc_workspace(desc, variant, True, dev)
    G = grads
    _check_grads(G, q, k, v, g, omega, r, out_dtype, ns, np_)
    _arg(workspace, "workspace", torch.uint8)
    st = getattr(lib(), name)(ctypes.byref(desc), _ptr(q), _ptr(k), _ptr(v), _ptr(g),
                              _ptr(omega), _ptr(r), _ptr(S0), _ptr(p0), _ptr(dO), _ptr(dST),
                              _ptr(dpT), _ptr(G["dq"]), _ptr(G["dk"]), _ptr(G["dv"]),
                              _ptr(G["dg"]), _ptr(G["domega"]), _ptr(G["dr"]),
                              _ptr(G.get("dS0")), _ptr(G.get("dp0")), _ptr(G.get("dmu")),
                              _ptr(workspace),
                              workspace.numel(), _stream(stream))
    _check(st, name)
    return grads


def kdn_diag_bwd(q, k, v, g, omega, r, S0, p0, dO, dST=None, dpT=None, *, chunk=0, mu=None,
                 scale=None, grads=None, want_state_grads=True, workspace=None, stream=None,
                 out_dtype=torch.float32, gates=KDN_GATES_POST,
                 r_min=R_MIN_DEFAULT):
    """Gradients of the Diagonal KDN forward.  Returns a dict dq, dk, dv, dg, domega, dr,
    and with want_state_grads dS0, dp0 and dmu [B,H] (the gradient with respect to mu)."""
    return _bwd("kdn_diag_bwd", 0, q, k, v, g, omega, r, S0, p0, dO, dST, dpT, chunk=chunk,
                mu=mu, scale=scale, grads=grads, want_state_grads=want_state_grads,
                workspace=workspace, stream=stream, out_dtype=out_dtype,
        gates=gates, r_min=r_min)


def kdn_iso_bwd(q, k, v, g, omega, r, S0, p0, dO, dST=None, dpT=None, *, chunk=0, mu=None,
                scale=None, grads=None, want_state_grads=True, workspace=None, stream=None,
                 out_dtype=torch.float32, gates=KDN_GATES_POST,
                 r_min=R_MIN_DEFAULT):
    """Gradients of the Isotropic KDN forward."""
    return _bwd("kdn_iso_bwd", 1, q, k, v, g, omega, r, S0, p0, dO, dST, dpT, chunk=chunk,
                mu=mu, scale=scale, grads=grads, want_state_grads=want_state_grads,
                workspace=workspace, stream=stream, out_dtype=out_dtype,
        gates=gates, r_min=r_min)


def saved_bytes(desc: kdn_desc_t, variant: int = 0) -> int:
    """Bytes of the saved backward context (0: the descriptor has no saved-context path)."""
    return int(lib().kdn_saved_bytes(ctypes.byref(desc), int(variant)))


def _fwd_save(name, variant, q, k, v, g, omega, r, S0, p0, *, mu, scale, o, ST, pT, saved,
              want_state, workspace, stream, out_dtype,
              gates=KDN_GATES_POST, r_min=R_MIN_DEFAULT):
    _check_inputs(variant, q, k, v, g, omega, r)
    desc = _desc_from(variant, q, v, g, chunk=0, mu=mu, scale=scale, out_dtype=out_dtype,
                      gates=gates, r_min=r_min)
    B, T, H, dk = q.shape
    dv = v.shape[-1]
    dev = q.device
    ns, np_ = _state_sizes(variant, q, v)
    _arg(S0, "S0", torch.float32, ns, required=False)
    _arg(p0, "p0", torch.float32, np_, required=False)
    if o is None:
        o = torch.empty(B, T, H, dv, dtype=out_dtype, device=dev)
    if want_state and ST is None:
        ST = torch.empty(B, H, dk, dv, dtype=torch.float32, device=dev)
    if want_state and pT is None:
        pT = torch.empty((B, H, dk) if variant == 0 else (B, H), dtype=torch.float32, device=dev)
    if saved is None:
        saved = torch.empty(max(saved_bytes(desc, variant), 256), dtype=torch.uint8, device=dev)
    if workspace is None:
        workspace = alloc_workspace(desc, variant, False, dev)
    _arg(o, "o", _torch_dtype(out_dtype), B * T * H * dv)
    _arg(ST, "ST", torch.float32, ns, required=False)
    _arg(pT, "pT", torch.float32, np_, required=False)
    _arg(saved, "saved", torch.uint8)
    _arg(workspace, "workspace", torch.uint8)
    st = getattr(lib(), name)(ctypes.byref(desc), _ptr(q), _ptr(k), _ptr(v), _ptr(g),
                              _ptr(omega), _ptr(r), _ptr(S0), _ptr(p0), _ptr(o), _ptr(ST),
                              _ptr(pT), _ptr(saved), saved.numel(), _ptr(workspace),
                              workspace.numel(), _stream(stream))
    _check(st, name)
    return o, ST, pT, saved


def kdn_diag_fwd_save(q, k, v, g, omega, r, S0=None, p0=None, *, mu=None, scale=None, o=None,
                      ST=None, pT=None, saved=None, want_state=True, workspace=None, stream=None,
                      out_dtype=torch.float32, gates=KDN_GATES_POST,
                 r_min=R_MIN_DEFAULT):
    """Diagonal KDN forward that also keeps the chunked backward's context.
    Returns (o, ST, pT, saved); pass `saved` to kdn_diag_bwd_saved."""
    return _fwd_save("kdn_diag_fwd_save", 0, q, k, v, g, omega, r, S0, p0, mu=mu, scale=scale,
                     o=o, ST=ST, pT=pT, saved=saved, want_state=want_state, workspace=workspace,
                     stream=stream, out_dtype=out_dtype,
        gates=gates, r_min=r_min)


def kdn_iso_fwd_save(q, k, v, g, omega, r, S0=None, p0=None, *, mu=None, scale=None, o=None,
                     ST=None, pT=None, saved=None, want_state=True, workspace=None, stream=None,
                     out_dtype=torch.float32, gates=KDN_GATES_POST,
                 r_min=R_MIN_DEFAULT):
    """Isotropic KDN forward that also keeps the chunked backward's context."""
    return _fwd_save("kdn_iso_fwd_save", 1, q, k, v, g, omega, r, S0, p0, mu=mu, scale=scale,
                     o=o, ST=ST, pT=pT, saved=saved, want_state=want_state, workspace=workspace,
                     stream=stream, out_dtype=out_dtype,
        gates=gates, r_min=r_min)


def _bwd_saved(name, variant, q, k, v, g, omega, r, saved, dO, dST, dpT, *, mu, scale, grads,
               want_state_grads, workspace, stream, out_dtype,
               gates=KDN_GATES_POST, r_min=R_MIN_DEFAULT):
    _check_inputs(variant, q, k, v, g, omega, r, dO)
    desc = _desc_from(variant, q, v, g, chunk=0, mu=mu, scale=scale, out_dtype=out_dtype,
                      gates=gates, r_min=r_min)
    B, T, H, dk = q.shape
    dv = v.shape[-1]
    dev = q.device
    ns, np_ = _state_sizes(variant, q, v)
    _arg(saved, "saved", torch.uint8)
    _arg(dST, "dST", torch.float32, ns, required=False)
    _arg(dpT, "dpT", torch.float32, np_, required=False)
    if grads is None:
        grads = {n: torch.empty(x.shape, dtype=out_dtype, device=dev) for n, x in
                 (("dq", q), ("dk", k), ("dv", v), ("dg", g), ("domega", omega), ("dr", r))}
        if want_state_grads:
            grads["dS0"] = torch.empty(B, H, dk, dv, dtype=torch.float32, device=dev)
            grads["dp0"] = torch.empty((B, H, dk) if variant == 0 else (B, H),
                                       dtype=torch.float32, device=dev)
            grads["dmu"] = torch.empty(B, H, dtype=torch.float32, device=dev)
    if workspace is None:
        workspace = alloc_workspace(desc, variant, False, dev)
    G = grads
    _check_grads(G, q, k, v, g, omega, r, out_dtype, ns, np_)
    _arg(workspace, "workspace", torch.uint8)
    st = getattr(lib(), name)(ctypes.byref(desc), _ptr(q), _ptr(k), _ptr(v), _ptr(g),
                              _ptr(omega), _ptr(r), _ptr(saved), saved.numel(), _ptr(dO),
                              _ptr(dST), _ptr(dpT), _ptr(G["dq"]), _ptr(G["dk"]),
                              _ptr(G["dv"]), _ptr(G["dg"]), _ptr(G["domega"]), _ptr(G["dr"]),
                              _ptr(G.get("dS0")), _ptr(G.get("dp0")), _ptr(G.get("dmu")),
                              _ptr(workspace),
                              workspace.numel(), _stream(stream))
    _check(st, name)
    return grads


def kdn_diag_bwd_saved(q, k, v, g, omega, r, saved, dO, dST=None, dpT=None, *, mu=None,
                       scale=None, grads=None, want_state_grads=True, workspace=None, stream=None,
                       out_dtype=torch.float32, gates=KDN_GATES_POST,
                 r_min=R_MIN_DEFAULT):
    """Gradients of the Diagonal KDN forward from the context kept by kdn_diag_fwd_save."""
    return _bwd_saved("kdn_diag_bwd_saved", 0, q, k, v, g, omega, r, saved, dO, dST, dpT, mu=mu,
                      scale=scale, grads=grads, want_state_grads=want_state_grads,
                      workspace=workspace, stream=stream, out_dtype=out_dtype,
        gates=gates, r_min=r_min)


def kdn_iso_bwd_saved(q, k, v, g, omega, r, saved, dO, dST=None, dpT=None, *, mu=None,
                      scale=None, grads=None, want_state_grads=True, workspace=None, stream=None,
                      out_dtype=torch.float32, gates=KDN_GATES_POST,
                 r_min=R_MIN_DEFAULT):
    """Gradients of the Isotropic KDN forward from the context kept by kdn_iso_fwd_save."""
    return _bwd_saved("kdn_iso_bwd_saved", 1, q, k, v, g, omega, r, saved, dO, dST, dpT, mu=mu,
                      scale=scale, grads=grads, want_state_grads=want_state_grads,
                      workspace=workspace, stream=stream, out_dtype=out_dtype,
        gates=gates, r_min=r_min)


def _beta_eff(name, variant, k, v, g, r, saved, *, out, stream, gates, r_min):
    desc = _desc_from(variant, k, v, g, chunk=0, mu=None, scale=None, out_dtype=torch.float32,
                      gates=gates, r_min=r_min)
    B, T, H, _ = k.shape
    _arg(k, "k")
    _arg(saved, "saved", torch.uint8)
    _arg(r, "r", k.dtype, B * T * H)
    if out is None:
        out = torch.empty(B, T, H, dtype=torch.float32, device=k.device)
    _arg(out, "out", torch.float32, B * T * H)
    st = getattr(lib(), name)(ctypes.byref(desc), _ptr(saved), ctypes.c_size_t(saved.numel()),
                              _ptr(r), _ptr(out), _stream(stream))
    _check(st, name)
    return out


def kdn_diag_beta_eff(k, v, g, r, saved, *, out=None, stream=None, gates=KDN_GATES_POST,
                      r_min=R_MIN_DEFAULT):
    """beta_eff = k_t^T kappa_t [B,T,H] (float32) from the context kdn_diag_fwd_save kept;
    k, v, g fix the descriptor, r is the forward's r."""
    return _beta_eff("kdn_diag_beta_eff", 0, k, v, g, r, saved, out=out, stream=stream,
                     gates=gates, r_min=r_min)


def kdn_iso_beta_eff(k, v, g, r, saved, *, out=None, stream=None, gates=KDN_GATES_POST,
                     r_min=R_MIN_DEFAULT):
    """beta_eff = beta_t |k_t|^2 [B,T,H] (float32) from the context kdn_iso_fwd_save kept."""
    return _beta_eff("kdn_iso_beta_eff", 1, k, v, g, r, saved, out=out, stream=stream,
                     gates=gates, r_min=r_min)


def _decode(name, variant, q, k, v, g, omega, r, S, p, *, mu, scale, o, stream, out_dtype,
            gates=KDN_GATES_POST, r_min=R_MIN_DEFAULT):
    _check_inputs(variant, q, k, v, g, omega, r, tokens=False)
    B, H, dk = q.shape
    dv = v.shape[-1]
    pcd = 1 if variant == 0 else int(g.dim() == 3)
    desc = make_desc(B, 1, H, dk, dv, q.dtype, mu=mu, scale=scale, decay_per_channel=pcd,
                     out_dtype=out_dtype,
        gates=gates, r_min=r_min)
    ns, np_ = _state_sizes(variant, q, v, tokens=False)
    _arg(S, "S", torch.float32, ns)
    _arg(p, "p", torch.float32, np_)
    if o is None:
        o = torch.empty(B, H, dv, dtype=out_dtype, device=q.device)
    _arg(o, "o", _torch_dtype(out_dtype), B * H * dv)
    st = getattr(lib(), name)(ctypes.byref(desc), _ptr(q), _ptr(k), _ptr(v), _ptr(g),
                              _ptr(omega), _ptr(r), _ptr(S), _ptr(p), _ptr(o), _stream(stream))
    _check(st, name)
    return o


def kdn_diag_decode_step(q, k, v, g, omega, r, S, p, *, mu=None, scale=None, o=None,
                         stream=None, out_dtype=torch.float32, gates=KDN_GATES_POST,
                 r_min=R_MIN_DEFAULT):
    """One Diagonal KDN token for every head, S [B,H,dk,dv] and p [B,H,dk] updated in place."""
    return _decode("kdn_diag_decode_step", 0, q, k, v, g, omega, r, S, p, mu=mu, scale=scale,
                   o=o, stream=stream, out_dtype=out_dtype,
        gates=gates, r_min=r_min)


def kdn_iso_decode_step(q, k, v, g, omega, r, S, p, *, mu=None, scale=None, o=None,
                        stream=None, out_dtype=torch.float32, gates=KDN_GATES_POST,
                 r_min=R_MIN_DEFAULT):
    """One Isotropic KDN token for every head; g [B,H,dk] or [B,H]; p [B,H] in place."""
    return _decode("kdn_iso_decode_step", 1, q, k, v, g, omega, r, S, p, mu=mu, scale=scale,
                   o=o, stream=stream, out_dtype=out_dtype,
        gates=gates, r_min=r_min)


def kdn_diag_fwd_noalloc(q, k, v, g, omega, r, S0=None, p0=None, *, o, ST=None, pT=None,
                         mu=None, scale=None, stream=None, gates=KDN_GATES_POST,
                         r_min=R_MIN_DEFAULT):
    """Diagonal KDN forward into caller-provided outputs, using the library's own
    fixed scratch array instead of a workspace, for callers that may not
    allocate device memory.  Problems needing more than
    KDN_NOALLOC_SCRATCH_BYTES of scratch are rejected.  Returns o."""
    _check_inputs(0, q, k, v, g, omega, r)
    _arg(o, "o")
    desc = _desc_from(0, q, v, g, chunk=0, mu=mu, scale=scale, out_dtype=o.dtype, gates=gates,
                      r_min=r_min)
    B, T, H, dk = q.shape
    ns, np_ = _state_sizes(0, q, v)
    _arg(o, "o", None, B * T * H * v.shape[-1])
    for t, n, m in ((S0, "S0", ns), (p0, "p0", np_), (ST, "ST", ns), (pT, "pT", np_)):
        _arg(t, n, torch.float32, m, required=False)
    st = lib().kdn_diag_fwd_noalloc(ctypes.byref(desc), _ptr(q), _ptr(k), _ptr(v), _ptr(g),
                                    _ptr(omega), _ptr(r), _ptr(S0), _ptr(p0), _ptr(o), _ptr(ST),
                                    _ptr(pT), _stream(stream))
    _check(st, "kdn_diag_fwd_noalloc")
    return o


def kdn_kernel_launches(desc: kdn_desc_t, variant: int, op: int) -> int:
    """Kernels one call launches (op 0 fwd, 1 bwd, 2 decode step)."""
    return int(lib().kdn_kernel_launches(ctypes.byref(desc), int(variant), int(op)))


def kdn_selftest_wait_timeout(workspace, stream=None) -> int:
    """Runs the device self-test of the bounded waits on ``workspace`` (asynchronous);
    kdn_get_device_status then reports KDN_ERR_TIMEOUT."""
    _arg(workspace, "workspace")
    return int(lib().kdn_selftest_wait_timeout(_ptr(workspace), _stream(stream)))


def kdn_get_device_status(workspace, stream=None) -> int:
    _arg(workspace, "workspace")
    return int(lib().kdn_get_device_status(_ptr(workspace), _stream(stream)))


def kdn_noalloc_device_status(stream=None) -> int:
    """Reads and clears the status word of the last kdn_diag_fwd_noalloc call."""
    return int(lib().kdn_noalloc_device_status(_stream(stream)))
