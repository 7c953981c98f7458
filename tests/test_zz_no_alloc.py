"""flex_linattn_bwd_noalloc, the backward for callers that cannot allocate device memory
and so pass no workspace (a framework whose pool owns the device memory, or a path that
must not call cudaMalloc/cudaFree).  Its scratch is a fixed array in the library's own
device memory, shared by every call.

Called through the C ABI with ctypes.  Two calls in a row, on different inputs, must each
match the fp64 oracle under the stated tolerances and the regular workspace-taking
flex_linattn_bwd within the same tolerance (the two run different kernels: this entry
point always takes the fp32 CUDA-core backward).  The array keeps the previous call's
contents, so the second call also checks that nothing of the first one leaks through.
This file is collected last on purpose.
"""
import ctypes

import numpy as np
import pytest
import torch

import oracle
from paper_2606_27748_gb300 import flexattn, workloads
from parity import assert_close, to_dev, to_host

pytestmark = pytest.mark.gpu

SCRATCH_FLOATS = 1 << 20  # the array's size, stated in include/flexattn.h


def _entry(lib):
    fn = lib.flex_linattn_bwd_noalloc
    vp = ctypes.c_void_p
    fn.argtypes = [ctypes.POINTER(flexattn.FlexShape)] + [vp] * 5 + [ctypes.c_int] + [vp] * 9
    fn.restype = ctypes.c_int
    return fn


@pytest.fixture(scope="module")
def lib():
    assert torch.cuda.is_available(), "GPU tests need CUDA"
    from paper_2606_27748_gb300 import build
    build.build()
    return flexattn.load()


def _p(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _call(fn, q, k, v, W1, W2, causal, out, den, dO):
    got = [torch.full_like(q, float("nan")), torch.full_like(k, float("nan")),
           torch.full_like(v, float("nan")), torch.full_like(W1, float("nan")),
           None if W2 is None else torch.full_like(W2, float("nan"))]
    shape = flexattn.shape_of(q, W1)
    rc = fn(ctypes.byref(shape), _p(q), _p(k), _p(v), _p(W1), _p(W2), int(causal),
            _p(out), _p(den), _p(dO), *[_p(t) for t in got],
            ctypes.c_void_p(torch.cuda.current_stream().cuda_stream))
    assert rc == flexattn.FLEX_OK, flexattn.strerror(rc)
    torch.cuda.synchronize()
    return got


def _check(w, got, ref, what):
    for name, g, r in zip(["dq", "dk", "dv", "dW1", "dW2"], got, ref):
        if r is None:
            assert g is None
            continue
        rh = r if isinstance(r, np.ndarray) else to_host(r)
        scale = float(np.sqrt(np.mean(rh * rh))) if name.startswith("dW") else 1.0
        assert_close(to_host(g), rh, w.dtype, f"{what} {name}", max_abs_scale=scale)


@pytest.mark.parametrize("w", [workloads.ORDERED[4], workloads.ORDERED[2], workloads.ORDERED[0]],
                         ids=["stationary", "nonstationary", "f32"])
@pytest.mark.parametrize("causal", [True, False])
def test_noalloc_matches_oracle_and_workspace_entry_point(lib, w, causal):
    fn = _entry(lib)
    for call, seed in enumerate((11, 12)):
        wr = w.replace(B=2, H=3, N=300, seed=seed, backward=True)
        ins = workloads.make_inputs(wr)
        q, k, v, dO = (to_dev(ins[n], w.dtype) for n in ("q", "k", "v", "dO"))
        W1, W2 = to_dev(ins["W1"], "f32"), to_dev(ins["W2"], "f32")
        out, den = flexattn.linattn_fwd(q, k, v, W1, W2, causal)
        n0 = flexattn.kernel_launches()
        got = _call(fn, q, k, v, W1, W2, causal, out, den, dO)
        assert flexattn.kernel_launches() - n0 == 2
        ref = oracle.bwd(ins["q"], ins["k"], ins["v"], ins["W1"], ins["W2"], causal, ins["dO"])
        _check(w, got, ref, f"call {call} vs oracle:")
        ws_ref = flexattn.linattn_bwd(q, k, v, W1, W2, causal, out, den, dO)
        _check(w, got, ws_ref, f"call {call} vs workspace entry point:")


def test_noalloc_size_limit_boundary(lib):
    """B * H * (Mc * d + 1) floats must fit the 2^20-float array: 255 sequences of
    Mc * d = 4096 fit (1,044,735 floats) and run correctly; 256 do not (1,048,832)."""
    fn = _entry(lib)
    w = workloads.ORDERED[1].replace(B=15, H=17, N=8, backward=True, seed=13)  # s, M 64, d 64
    assert w.B * w.H * (w.M * w.d + 1) <= SCRATCH_FLOATS
    ins = workloads.make_inputs(w)
    q, k, v, dO = (to_dev(ins[n], w.dtype) for n in ("q", "k", "v", "dO"))
    W1 = to_dev(ins["W1"], "f32")
    out, den = flexattn.linattn_fwd(q, k, v, W1, None, True)
    got = _call(fn, q, k, v, W1, None, True, out, den, dO)
    ref = oracle.bwd(ins["q"], ins["k"], ins["v"], ins["W1"], None, True, ins["dO"])
    _check(w, got, ref, "255 sequences:")

    over = flexattn.FlexShape(16, 16, 8, 64, 64, flexattn.FLEX_BF16)
    assert 16 * 16 * (64 * 64 + 1) > SCRATCH_FLOATS
    p = ctypes.c_void_p(1 << 20)  # never dereferenced: the size check fails first
    rc = fn(ctypes.byref(over), p, p, p, p, None, 1, p, p, p, p, p, p, p, None, None)
    assert rc == flexattn.FLEX_EWORKSPACE
    # far beyond: 8 x 16 sequences x 2M = 256 rows x d = 64 -> 2^21 floats
    far = flexattn.FlexShape(8, 16, 128, 64, 128, flexattn.FLEX_BF16)
    rc = fn(ctypes.byref(far), p, p, p, p, p, 1, p, p, p, p, p, p, p, p, None)
    assert rc == flexattn.FLEX_EWORKSPACE
