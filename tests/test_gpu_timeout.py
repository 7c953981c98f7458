"""Failure detection on the device: a bounded wait that runs out.

Every wait of the tensor-core kernels is bounded; when one gives up, the CTA sets its
abort flag, every other wait returns, the kernel frees its tensor memory and exits, and the
workspace records FLEX_ETIMEOUT for flex_check_status.  Here a wait is made to run out on
purpose without any fault: flex_debug_stall asks each CTA of the causal forward to wait,
with a limit of a few microseconds, on an mbarrier that nothing arrives on, before it
issues any copy or tensor-core operation.  The test checks the status, that nothing was
written, and that the same stream and workspace then run a correct forward.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2606_27748_gb300 import flexattn, workloads
from parity import assert_close, to_dev, to_host

pytestmark = pytest.mark.gpu

WL = workloads.ORDERED


@pytest.fixture(scope="module", autouse=True)
def library():
    assert torch.cuda.is_available(), "GPU tests need CUDA"
    from paper_2606_27748_gb300 import build
    build.build()
    flexattn.load()


@pytest.mark.parametrize("w", [WL[1], WL[2]], ids=["single-CTA", "cluster-pair"])
def test_bounded_wait_runs_out_and_stream_stays_usable(w):
    ws_ = w.replace(B=1, H=2, N=700)  # several chunks; 2-3 segments per sequence
    ins = workloads.make_inputs(ws_)
    q, k, v = (to_dev(ins[n], w.dtype) for n in "qkv")
    W1, W2 = to_dev(ins["W1"], "f32"), to_dev(ins["W2"], "f32")
    ws = flexattn.workspace(flexattn.shape_of(q, W1), True, False)
    out = torch.full_like(q, float("nan"))
    den = torch.full(q.shape[:3], float("nan"), dtype=torch.float32, device=q.device)

    flexattn.debug_stall(ws, 20000)  # ~10 us at 2 GHz
    flexattn.linattn_fwd(q, k, v, W1, W2, True, out=out, den=den, ws=ws)
    with pytest.raises(flexattn.FlexError) as e:
        flexattn.check_status(ws)
    assert e.value.status == flexattn.FLEX_ETIMEOUT
    assert torch.isnan(out.float()).all() and torch.isnan(den).all()  # nothing issued

    flexattn.debug_stall(ws, 0)
    flexattn.linattn_fwd(q, k, v, W1, W2, True, out=out, den=den, ws=ws)
    flexattn.check_status(ws)  # FLEX_OK: the status was cleared by the first check
    ro, rd = oracle.fwd(ins["q"], ins["k"], ins["v"], ins["W1"], ins["W2"], True)
    assert_close(to_host(out), ro, w.dtype, "out")
    assert_close(to_host(den), rd, w.dtype, "den", max_abs_scale=float(np.abs(rd).max()))
