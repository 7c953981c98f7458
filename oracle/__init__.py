"""fp64 CPU oracle for Flexformer random-Fourier-feature linear attention.

TEST INFRASTRUCTURE ONLY.  Only ``tests/``, ``__graft_entry__.smoke()`` and the CPU
baseline leg of ``bench.py`` may import this package.  The product path (the CUDA library
and its Python binding) never imports, links or executes anything here, and this package
imports nothing from the product path.

Contents
  * ``flex_oracle.c`` -- the linear form (Sec. 2.2, Eq. linear att) with the stationary
    (Eq. phi_n, Flexformer_s) and nonstationary (Eq. phi_non, Flexformer_n) feature maps,
    forward and analytic backward, in plain fp64 C loops.  Loaded here through ctypes.
  * ``brute.py`` -- the explicit N x N kernel-matrix form of Eq. (attention) with
    sim(q, k) = phi(q) . phi(k) (Eq. kernel), written independently in numpy, and the
    distillation loss written with explicit matrices.

Every function takes and returns float64 numpy arrays in the layouts
q, k, v, out: [B, H, N, d];  W1, W2: [H, M, d];  den: [B, H, N];  phi: [B, H, N, 2M].
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
SOURCE = os.path.join(_HERE, "flex_oracle.c")
BUILD_DIR = os.path.join(_HERE, "_build")
LIBRARY = os.path.join(BUILD_DIR, "libflex_oracle.so")

_lock = threading.Lock()
_lib = None


def compile_library(source_text: str | None = None, out_path: str = LIBRARY) -> str:
    """Compile the C oracle (or a modified copy of its source text) into a shared library.

    Plain gcc, -O2, no fast-math: the oracle keeps IEEE fp64 semantics.
    """
    os.makedirs(os.path.dirname(out_path), exist_ok=True)
    src = SOURCE
    if source_text is not None:
        src = out_path[:-3] + ".c"
        with open(src, "w") as f:
            f.write(source_text)
    tmp = out_path + f".tmp{os.getpid()}"
    subprocess.run(["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-pthread", src, "-o", tmp,
                    "-lm"], check=True)
    os.replace(tmp, out_path)
    return out_path


def _stale() -> bool:
    return (not os.path.exists(LIBRARY)
            or os.path.getmtime(LIBRARY) < os.path.getmtime(SOURCE))


class Oracle:
    """ctypes view of one compiled copy of ``flex_oracle.c``."""

    def __init__(self, path: str):
        lib = ctypes.CDLL(path)
        dp = ctypes.POINTER(ctypes.c_double)
        i = ctypes.c_int
        lib.oracle_featmap.argtypes = [i, i, i, i, i, dp, dp, dp, dp]
        lib.oracle_featmap_sumform.argtypes = [i, i, i, i, i, dp, dp, dp, dp]
        lib.oracle_linattn_fwd.argtypes = [i, i, i, i, i, dp, dp, dp, dp, dp, dp, i, dp, dp, i]
        lib.oracle_linattn_bwd.argtypes = [i, i, i, i, i, dp, dp, dp, dp, dp, dp, i, dp, dp, dp,
                                           dp, dp, dp, dp, i]
        lib.oracle_linattn_decode.argtypes = [i, i, i, i, dp, dp, dp, dp, dp, dp, dp, dp, dp,
                                              dp]
        lib.oracle_awd.argtypes = [i, i, i, i, i, dp, dp, dp, dp, dp, i, dp]
        lib.oracle_awd_bwd.argtypes = [i, i, i, i, i, dp, dp, dp, dp, dp, i, dp, dp, dp, dp]
        for fn in (lib.oracle_featmap, lib.oracle_featmap_sumform, lib.oracle_linattn_fwd,
                   lib.oracle_linattn_bwd, lib.oracle_linattn_decode, lib.oracle_awd,
                   lib.oracle_awd_bwd):
            fn.restype = ctypes.c_int
        self._lib = lib
        self.path = path

    @staticmethod
    def _p(a):
        if a is None:
            return None
        return a.ctypes.data_as(ctypes.POINTER(ctypes.c_double))

    @staticmethod
    def _f64(a):
        return None if a is None else np.ascontiguousarray(a, dtype=np.float64)

    def featmap(self, x, W1, W2=None):
        """phi(x) for x [B, H, N, d] with per-head frequencies [H, M, d] -> [B, H, N, 2M]."""
        x, W1, W2 = self._f64(x), self._f64(W1), self._f64(W2)
        B, H, N, d = x.shape
        M = W1.shape[1]
        phi = np.empty((B, H, N, 2 * M))
        rc = self._lib.oracle_featmap(B, H, N, d, M, self._p(x), self._p(W1), self._p(W2),
                                      self._p(phi))
        if rc != 0:
            raise ValueError("oracle_featmap: bad shape")
        return phi

    def featmap_sumform(self, x, W1, W2):
        """Nonstationary phi(x) in the unsimplified Monte Carlo form of Eq. (phi_non)."""
        x, W1, W2 = self._f64(x), self._f64(W1), self._f64(W2)
        B, H, N, d = x.shape
        M = W1.shape[1]
        phi = np.empty((B, H, N, 2 * M))
        rc = self._lib.oracle_featmap_sumform(B, H, N, d, M, self._p(x), self._p(W1),
                                              self._p(W2), self._p(phi))
        if rc != 0:
            raise ValueError("oracle_featmap_sumform: bad shape")
        return phi

    def fwd(self, q, k, v, W1, W2=None, causal=True, nthreads=None, tau=None):
        """(out [B, H, N, d], den [B, H, N]) of Eq. (linear att); tau [H]: the norm
        prefactor of Sec. 3.2 (a key weight; den excludes the query's factor)."""
        q, k, v, W1, W2, tau = (self._f64(a) for a in (q, k, v, W1, W2, tau))
        B, H, N, d = q.shape
        M = W1.shape[1]
        out = np.empty_like(q)
        den = np.empty((B, H, N))
        nt = nthreads or os.cpu_count() or 1
        rc = self._lib.oracle_linattn_fwd(B, H, N, d, M, self._p(q), self._p(k), self._p(v),
                                          self._p(W1), self._p(W2), self._p(tau),
                                          int(bool(causal)), self._p(out), self._p(den), nt)
        if rc != 0:
            raise ValueError("oracle_linattn_fwd: bad shape")
        return out, den

    def bwd(self, q, k, v, W1, W2, causal, dout, nthreads=None, tau=None):
        """Gradients (dq, dk, dv, dW1, dW2) of L = sum(dout * out); dW2 is None if W2 is.
        With tau [H] (the norm prefactor) a sixth value, dtau [H], follows."""
        q, k, v, W1, W2, dout, tau = (self._f64(a) for a in (q, k, v, W1, W2, dout, tau))
        B, H, N, d = q.shape
        M = W1.shape[1]
        dq, dk, dv = np.empty_like(q), np.empty_like(q), np.empty_like(q)
        dW1 = np.empty_like(W1)
        dW2 = None if W2 is None else np.empty_like(W2)
        dtau = None if tau is None else np.empty(H)
        nt = nthreads or os.cpu_count() or 1
        rc = self._lib.oracle_linattn_bwd(B, H, N, d, M, self._p(q), self._p(k), self._p(v),
                                          self._p(W1), self._p(W2), self._p(tau),
                                          int(bool(causal)), self._p(dout), self._p(dq),
                                          self._p(dk), self._p(dv), self._p(dW1), self._p(dW2),
                                          self._p(dtau), nt)
        if rc != 0:
            raise ValueError("oracle_linattn_bwd: bad shape")
        if tau is None:
            return dq, dk, dv, dW1, dW2
        return dq, dk, dv, dW1, dW2, dtau

    def decode(self, q, k, v, W1, W2, S, z, tau=None):
        """One causal decode step (Eq. linear att as running sums, inclusive of the new
        token): q, k, v [B, H, d]; state S [B, H, 2M, d], z [B, H, 2M] (not modified);
        tau [H] or None.  Returns (out [B, H, d], den [B, H], S', z')."""
        q, k, v, W1, W2, tau = (self._f64(a) for a in (q, k, v, W1, W2, tau))
        S = np.array(S, dtype=np.float64, copy=True, order="C")
        z = np.array(z, dtype=np.float64, copy=True, order="C")
        B, H, d = q.shape
        M = W1.shape[1]
        out = np.empty_like(q)
        den = np.empty((B, H))
        rc = self._lib.oracle_linattn_decode(B, H, d, M, self._p(q), self._p(k), self._p(v),
                                             self._p(W1), self._p(W2), self._p(tau), self._p(S),
                                             self._p(z), self._p(out), self._p(den))
        if rc != 0:
            raise ValueError("oracle_linattn_decode: bad shape")
        return out, den, S, z


    def awd(self, q, k, W1, W2=None, causal=False, tau=None):
        """Attention-weight distillation loss of every sequence, [B, H]: the cross-entropy
        of the kernel's normalised weights against softmax(q k^T / sqrt(d)), averaged over
        the queries (entries with a non-positive kernel estimate count log 1e-6)."""
        q, k, W1, W2, tau = (self._f64(a) for a in (q, k, W1, W2, tau))
        B, H, N, d = q.shape
        M = W1.shape[1]
        loss = np.empty((B, H))
        rc = self._lib.oracle_awd(B, H, N, d, M, self._p(q), self._p(k), self._p(W1),
                                  self._p(W2), self._p(tau), int(bool(causal)), self._p(loss))
        if rc != 0:
            raise ValueError("oracle_awd: bad shape")
        return loss

    def awd_bwd(self, q, k, W1, W2=None, causal=False, tau=None, dloss=None):
        """Gradient of sum_{b,h} dloss[b, h] * awd(...)[b, h] with respect to the kernel's
        parameters: (dW1 [H, M, d], dW2 [H, M, d] or None, dtau [H] or None).  dloss
        defaults to ones."""
        q, k, W1, W2, tau = (self._f64(a) for a in (q, k, W1, W2, tau))
        B, H, N, d = q.shape
        M = W1.shape[1]
        dl = self._f64(np.ones((B, H)) if dloss is None else np.broadcast_to(dloss, (B, H)))
        dW1 = np.empty_like(W1)
        dW2 = None if W2 is None else np.empty_like(W2)
        dtau = None if tau is None else np.empty(H)
        rc = self._lib.oracle_awd_bwd(B, H, N, d, M, self._p(q), self._p(k), self._p(W1),
                                      self._p(W2), self._p(tau), int(bool(causal)),
                                      self._p(dl), self._p(dW1), self._p(dW2), self._p(dtau))
        if rc != 0:
            raise ValueError("oracle_awd_bwd: bad shape")
        return dW1, dW2, dtau


def load() -> Oracle:
    """The oracle built from ``flex_oracle.c`` (compiled on first use if needed)."""
    global _lib
    with _lock:
        if _lib is None:
            if _stale():
                compile_library()
            _lib = Oracle(LIBRARY)
        return _lib


def featmap(x, W1, W2=None):
    return load().featmap(x, W1, W2)


def fwd(q, k, v, W1, W2=None, causal=True, nthreads=None, tau=None):
    return load().fwd(q, k, v, W1, W2, causal, nthreads, tau)


def bwd(q, k, v, W1, W2, causal, dout, nthreads=None, tau=None):
    return load().bwd(q, k, v, W1, W2, causal, dout, nthreads, tau)


def decode(q, k, v, W1, W2, S, z, tau=None):
    return load().decode(q, k, v, W1, W2, S, z, tau)


def awd(q, k, W1, W2=None, causal=False, tau=None):
    return load().awd(q, k, W1, W2, causal, tau)


def awd_bwd(q, k, W1, W2=None, causal=False, tau=None, dloss=None):
    return load().awd_bwd(q, k, W1, W2, causal, tau, dloss)
