"""flex_linattn_bwd_noalloc (the backward for callers that cannot allocate device memory
and so pass no workspace) against the regular workspace-taking flex_linattn_bwd.

Called through the C ABI with ctypes.  Two calls in a row, on different inputs, must
each match the regular entry point; the fixed scratch array is shared by all calls and
keeps the previous call's contents, so the second call also checks that nothing of the
first one leaks through.  This file is collected last on purpose.
"""
import ctypes

import numpy as np
import pytest
import torch

from paper_2606_27748_gb300 import flexattn, workloads
from parity import assert_close, to_dev, to_host

pytestmark = pytest.mark.gpu


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


@pytest.mark.parametrize("w", [workloads.ORDERED[4], workloads.ORDERED[2]],
                         ids=["stationary", "nonstationary"])
@pytest.mark.parametrize("causal", [True, False])
def test_noalloc_matches_workspace_entry_point(lib, w, causal):
    fn = _entry(lib)
    for call, seed in enumerate((11, 12)):
        wr = w.replace(B=2, H=3, N=300, seed=seed, backward=True)
        ins = workloads.make_inputs(wr)
        q, k, v, dO = (to_dev(ins[n], w.dtype) for n in ("q", "k", "v", "dO"))
        W1, W2 = to_dev(ins["W1"], "f32"), to_dev(ins["W2"], "f32")
        out, den = flexattn.linattn_fwd(q, k, v, W1, W2, causal)
        ref = flexattn.linattn_bwd(q, k, v, W1, W2, causal, out, den, dO)
        got = [torch.full_like(q, float("nan")), torch.full_like(k, float("nan")),
               torch.full_like(v, float("nan")), torch.full_like(W1, float("nan")),
               None if W2 is None else torch.full_like(W2, float("nan"))]
        shape = flexattn.shape_of(q, W1)
        rc = fn(ctypes.byref(shape), _p(q), _p(k), _p(v), _p(W1), _p(W2), int(causal),
                _p(out), _p(den), _p(dO), *[_p(t) for t in got],
                ctypes.c_void_p(torch.cuda.current_stream().cuda_stream))
        assert rc == flexattn.FLEX_OK, flexattn.strerror(rc)
        torch.cuda.synchronize()
        for name, g, r in zip(["dq", "dk", "dv", "dW1", "dW2"], got, ref):
            if r is None:
                assert g is None
                continue
            rh = to_host(r)
            scale = float(np.sqrt(np.mean(rh * rh))) if name.startswith("dW") else 1.0
            assert_close(to_host(g), rh, w.dtype, f"call {call} {name}", max_abs_scale=scale)


def test_noalloc_refuses_sizes_beyond_its_scratch(lib):
    fn = _entry(lib)
    # 8 * 16 sequences x 2M = 256 partial rows x d = 64 -> 2^21 floats > 2^20 available
    shape = flexattn.FlexShape(8, 16, 128, 64, 128, flexattn.FLEX_BF16)
    p = ctypes.c_void_p(1 << 20)  # never dereferenced: the size check fails first
    rc = fn(ctypes.byref(shape), p, p, p, p, p, 1, p, p, p, p, p, p, p, p, None)
    assert rc == flexattn.FLEX_EWORKSPACE
