"""Thin ctypes binding of ``libflexattn.so`` (C ABI: ``include/flexattn.h``).

Argument marshalling only: every step of the computation runs in the library's CUDA
kernels.  Tensors are torch CUDA tensors (torch supplies device memory and the current
stream); they are passed to the library as raw device pointers.  There is no CPU path:
if the library is missing or fails to load, every call raises.
"""
from __future__ import annotations

import ctypes
import os
import threading

import torch

_PKG = os.path.dirname(os.path.abspath(__file__))
LIBRARY = os.path.join(_PKG, "libflexattn.so")

FLEX_F32, FLEX_BF16 = 0, 1
FLEX_OK, FLEX_EINVAL, FLEX_EUNSUPPORTED, FLEX_EWORKSPACE, FLEX_ECUDA, FLEX_ETIMEOUT = (
    0, -1, -2, -3, -4, -5)

EXPORTS = ("flex_strerror", "flex_workspace_bytes", "flex_featmap", "flex_linattn_fwd",
           "flex_linattn_bwd", "flex_decode_workspace_bytes", "flex_linattn_decode",
           "flex_awd_workspace_bytes", "flex_awd_loss", "flex_awd_bwd_workspace_bytes",
           "flex_awd_loss_bwd", "flex_kernel_launches", "flex_check_status",
           "flex_debug_stall")


class FlexShape(ctypes.Structure):
    _fields_ = [("B", ctypes.c_int), ("H", ctypes.c_int), ("N", ctypes.c_int),
                ("d", ctypes.c_int), ("M", ctypes.c_int), ("dtype", ctypes.c_int)]


class FlexError(RuntimeError):
    def __init__(self, status: int, what: str):
        self.status = status
        super().__init__(f"{what}: {strerror(status)} ({status})")


_lock = threading.Lock()
_lib = None


def load(path: str = LIBRARY) -> ctypes.CDLL:
    """Open the library (once).  Raises if it has not been built."""
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        if not os.path.exists(path):
            raise RuntimeError(f"{path} is missing: build it with "
                               "`python -m paper_2606_27748_gb300.build`")
        lib = ctypes.CDLL(path)
        vp, sz, ip = ctypes.c_void_p, ctypes.c_size_t, ctypes.c_int
        shp = ctypes.POINTER(FlexShape)
        lib.flex_strerror.argtypes = [ip]
        lib.flex_strerror.restype = ctypes.c_char_p
        lib.flex_workspace_bytes.argtypes = [shp, ip, ip]
        lib.flex_workspace_bytes.restype = sz
        lib.flex_featmap.argtypes = [shp, vp, vp, vp, vp, vp]
        lib.flex_linattn_fwd.argtypes = [shp, vp, vp, vp, vp, vp, vp, ip, vp, vp, vp, sz, vp]
        lib.flex_linattn_bwd.argtypes = [shp, vp, vp, vp, vp, vp, vp, ip, vp, vp, vp, vp, vp,
                                         vp, vp, vp, vp, vp, sz, vp]
        lib.flex_decode_workspace_bytes.argtypes = [shp]
        lib.flex_decode_workspace_bytes.restype = sz
        lib.flex_linattn_decode.argtypes = [shp, vp, vp, vp, vp, vp, vp, vp, vp, vp, vp, vp,
                                            sz, vp]
        lib.flex_awd_workspace_bytes.argtypes = [shp]
        lib.flex_awd_workspace_bytes.restype = sz
        lib.flex_awd_loss.argtypes = [shp, vp, vp, vp, vp, vp, ip, vp, vp, sz, vp]
        lib.flex_awd_bwd_workspace_bytes.argtypes = [shp]
        lib.flex_awd_bwd_workspace_bytes.restype = sz
        lib.flex_awd_loss_bwd.argtypes = [shp, vp, vp, vp, vp, vp, ip, vp, vp, vp, vp, vp, vp,
                                          sz, vp]
        lib.flex_check_status.argtypes = [vp, vp]
        lib.flex_debug_stall.argtypes = [vp, sz, ip, vp]
        lib.flex_kernel_launches.argtypes = []
        lib.flex_kernel_launches.restype = ctypes.c_ulonglong
        for fn in (lib.flex_featmap, lib.flex_linattn_fwd, lib.flex_linattn_bwd,
                   lib.flex_linattn_decode, lib.flex_awd_loss, lib.flex_awd_loss_bwd,
                   lib.flex_check_status, lib.flex_debug_stall):
            fn.restype = ip
        _lib = lib
        return lib


def strerror(status: int) -> str:
    return load().flex_strerror(int(status)).decode()


def _dtype_code(t: torch.Tensor) -> int:
    if t.dtype == torch.float32:
        return FLEX_F32
    if t.dtype == torch.bfloat16:
        return FLEX_BF16
    raise TypeError(f"unsupported dtype {t.dtype}")


def _ptr(t):
    if t is None:
        return None
    if not t.is_cuda or not t.is_contiguous():
        raise ValueError("tensors must be contiguous CUDA tensors")
    return ctypes.c_void_p(t.data_ptr())


def _stream(stream):
    s = torch.cuda.current_stream() if stream is None else stream
    return ctypes.c_void_p(s.cuda_stream)


def shape_of(x: torch.Tensor, W1: torch.Tensor) -> FlexShape:
    B, H, N, d = x.shape
    return FlexShape(B, H, N, d, W1.shape[1], _dtype_code(x))


def workspace_bytes(shape: FlexShape, causal: bool, backward: bool) -> int:
    return int(load().flex_workspace_bytes(ctypes.byref(shape), int(causal), int(backward)))


def workspace(shape: FlexShape, causal: bool, backward: bool, device=None) -> torch.Tensor:
    """A caller-owned, zero-filled workspace (torch allocates it; the library never does)."""
    n = workspace_bytes(shape, causal, backward)
    if n == 0:
        raise FlexError(FLEX_EUNSUPPORTED, "flex_workspace_bytes")
    return torch.zeros(n, dtype=torch.uint8, device=device or "cuda")


def kernel_launches() -> int:
    """Cumulative count of kernels the library has enqueued in this process."""
    return int(load().flex_kernel_launches())


def _check(rc: int, what: str):
    if rc != FLEX_OK:
        raise FlexError(rc, what)


def featmap(x, W1, W2=None, phi=None, stream=None):
    """phi(x) [B, H, N, 2M] (Eq. phi_n, or Eq. phi_non when W2 is given)."""
    shape = shape_of(x, W1)
    if phi is None:
        phi = torch.empty(*x.shape[:3], 2 * shape.M, dtype=x.dtype, device=x.device)
    _check(load().flex_featmap(ctypes.byref(shape), _ptr(x), _ptr(W1), _ptr(W2), _ptr(phi),
                               _stream(stream)), "flex_featmap")
    return phi


def linattn_fwd(q, k, v, W1, W2=None, causal=True, out=None, den=None, ws=None,
                want_den=True, stream=None, tau=None):
    """(out, den) of Eq. (linear att); den is None unless want_den or given.  tau [H] fp32:
    the norm prefactor exp(|x|^2 / exp(tau)) (a key weight; den excludes the query's)."""
    shape = shape_of(q, W1)
    if out is None:
        out = torch.empty_like(q)
    if den is None and want_den:
        den = torch.empty(q.shape[:3], dtype=torch.float32, device=q.device)
    if ws is None:
        ws = workspace(shape, causal, False, q.device)
    _check(load().flex_linattn_fwd(ctypes.byref(shape), _ptr(q), _ptr(k), _ptr(v), _ptr(W1),
                                   _ptr(W2), _ptr(tau), int(bool(causal)), _ptr(out), _ptr(den),
                                   _ptr(ws), ws.numel(), _stream(stream)), "flex_linattn_fwd")
    return out, den


def linattn_bwd(q, k, v, W1, W2, causal, out, den, dout, dq=None, dk=None, dv=None,
                dW1=None, dW2=None, ws=None, stream=None, tau=None, dtau=None):
    """(dq, dk, dv, dW1, dW2) of L = sum(dout * out); dW2 is None when W2 is.  With tau
    (the forward's norm prefactor) a sixth value, dtau [H], follows."""
    shape = shape_of(q, W1)
    dq = torch.empty_like(q) if dq is None else dq
    dk = torch.empty_like(k) if dk is None else dk
    dv = torch.empty_like(v) if dv is None else dv
    dW1 = torch.empty_like(W1) if dW1 is None else dW1
    if W2 is not None and dW2 is None:
        dW2 = torch.empty_like(W2)
    if tau is not None and dtau is None:
        dtau = torch.empty_like(tau)
    if ws is None:
        ws = workspace(shape, causal, True, q.device)
    _check(load().flex_linattn_bwd(ctypes.byref(shape), _ptr(q), _ptr(k), _ptr(v), _ptr(W1),
                                   _ptr(W2), _ptr(tau), int(bool(causal)), _ptr(out), _ptr(den),
                                   _ptr(dout), _ptr(dq), _ptr(dk), _ptr(dv), _ptr(dW1),
                                   _ptr(dW2), _ptr(dtau), _ptr(ws), ws.numel(), _stream(stream)),
           "flex_linattn_bwd")
    if tau is None:
        return dq, dk, dv, dW1, dW2
    return dq, dk, dv, dW1, dW2, dtau


def decode_state(B, H, M, d, device=None):
    """A zero state (S [B, H, 2M, d], z [B, H, 2M], fp32) for flex_linattn_decode."""
    dev = device or "cuda"
    return (torch.zeros(B, H, 2 * M, d, dtype=torch.float32, device=dev),
            torch.zeros(B, H, 2 * M, dtype=torch.float32, device=dev))


def decode_workspace(B, H, M, d, device=None) -> torch.Tensor:
    """A caller-owned workspace for flex_linattn_decode (allocate once per serving loop)."""
    n = int(load().flex_decode_workspace_bytes(ctypes.byref(FlexShape(B, H, 1, d, M, 0))))
    if n == 0:
        raise FlexError(FLEX_EINVAL, "flex_decode_workspace_bytes")
    return torch.zeros(n, dtype=torch.uint8, device=device or "cuda")


def linattn_decode(q, k, v, W1, W2, S, z, out=None, den=None, want_den=True, ws=None,
                   stream=None, tau=None):
    """One recurrent decode step: q, k, v [B, H, d] (one new token per sequence); the fp32
    state (S, z) is updated in place.  Returns (out [B, H, d], den [B, H] or None)."""
    B, H, d = q.shape
    shape = FlexShape(B, H, 1, d, W1.shape[1], _dtype_code(q))
    if out is None:
        out = torch.empty_like(q)
    if den is None and want_den:
        den = torch.empty(B, H, dtype=torch.float32, device=q.device)
    if ws is None:
        ws = decode_workspace(B, H, W1.shape[1], d, q.device)
    _check(load().flex_linattn_decode(ctypes.byref(shape), _ptr(q), _ptr(k), _ptr(v),
                                      _ptr(W1), _ptr(W2), _ptr(tau), _ptr(S), _ptr(z), _ptr(out),
                                      _ptr(den), _ptr(ws), ws.numel(), _stream(stream)),
           "flex_linattn_decode")
    return out, den


def awd_workspace(shape: FlexShape, device=None) -> torch.Tensor:
    """A caller-owned workspace for flex_awd_loss."""
    n = int(load().flex_awd_workspace_bytes(ctypes.byref(shape)))
    if n == 0:
        raise FlexError(FLEX_EUNSUPPORTED, "flex_awd_workspace_bytes")
    return torch.zeros(n, dtype=torch.uint8, device=device or "cuda")


def awd_loss(q, k, W1, W2=None, causal=False, tau=None, loss=None, ws=None, stream=None):
    """Attention-weight distillation loss of every sequence, [B, H] fp32: the cross-entropy
    of this kernel's normalised attention weights against softmax(q k^T / sqrt(d))."""
    shape = shape_of(q, W1)
    if loss is None:
        loss = torch.empty(q.shape[:2], dtype=torch.float32, device=q.device)
    if ws is None:
        ws = awd_workspace(shape, q.device)
    _check(load().flex_awd_loss(ctypes.byref(shape), _ptr(q), _ptr(k), _ptr(W1), _ptr(W2),
                                _ptr(tau), int(bool(causal)), _ptr(loss), _ptr(ws),
                                ws.numel(), _stream(stream)), "flex_awd_loss")
    return loss


def awd_bwd_workspace(shape: FlexShape, device=None) -> torch.Tensor:
    """A caller-owned workspace for flex_awd_loss_bwd."""
    n = int(load().flex_awd_bwd_workspace_bytes(ctypes.byref(shape)))
    if n == 0:
        raise FlexError(FLEX_EUNSUPPORTED, "flex_awd_bwd_workspace_bytes")
    return torch.zeros(n, dtype=torch.uint8, device=device or "cuda")


def awd_loss_bwd(q, k, W1, W2=None, causal=False, tau=None, dloss=None, loss=None,
                 dW1=None, dW2=None, dtau=None, ws=None, stream=None, want_loss=True):
    """Distillation loss [B, H] (None unless want_loss) and its gradient with respect to the
    kernel's parameters, weighted by dloss [B, H] (default ones): (loss, dW1, dW2, dtau);
    dW2 is None without W2, dtau None without tau."""
    shape = shape_of(q, W1)
    dev = q.device
    if dloss is None:
        dloss = torch.ones(q.shape[:2], dtype=torch.float32, device=dev)
    if want_loss and loss is None:
        loss = torch.empty(q.shape[:2], dtype=torch.float32, device=dev)
    if dW1 is None:
        dW1 = torch.empty_like(W1)
    if W2 is not None and dW2 is None:
        dW2 = torch.empty_like(W2)
    if tau is not None and dtau is None:
        dtau = torch.empty_like(tau)
    if ws is None:
        ws = awd_bwd_workspace(shape, dev)
    _check(load().flex_awd_loss_bwd(ctypes.byref(shape), _ptr(q), _ptr(k), _ptr(W1), _ptr(W2),
                                    _ptr(tau), int(bool(causal)), _ptr(dloss),
                                    _ptr(loss if want_loss else None), _ptr(dW1),
                                    _ptr(dW2 if W2 is not None else None),
                                    _ptr(dtau if tau is not None else None), _ptr(ws),
                                    ws.numel(), _stream(stream)), "flex_awd_loss_bwd")
    return (loss if want_loss else None), dW1, (dW2 if W2 is not None else None), (
        dtau if tau is not None else None)


def check_status(ws, stream=None):
    """Synchronise and raise if a kernel that used `ws` gave up on a bounded wait."""
    _check(load().flex_check_status(_ptr(ws), _stream(stream)), "flex_check_status")


def debug_stall(ws, cycles: int, stream=None):
    """Diagnostic of the bounded waits: while `cycles` > 0, the causal tensor-core forward
    run with workspace `ws` gives up after a wait of at most `cycles` clocks that nothing
    ends, before doing any work (FLEX_ETIMEOUT through check_status).  0 restores it."""
    _check(load().flex_debug_stall(_ptr(ws), ws.numel(), int(cycles), _stream(stream)),
           "flex_debug_stall")
