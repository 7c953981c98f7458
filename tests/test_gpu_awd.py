"""Attention-weight distillation loss on the GPU against the fp64 oracle: both variants,
M = 64 and 128, causal and not, with and without the norm prefactor, sizes that leave a
ragged last block; a case with non-positive kernel estimates; launch counts and bit-exact
repeatability."""
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


def _cases():
    # (base workload, M, causal, tau, N)
    return [(WL[3], 64, False, False, 300), (WL[3], 64, True, False, 300),
            (WL[2], 128, False, True, 520), (WL[2], 128, True, True, 257),
            (WL[1], 64, False, True, 129), (WL[1], 128, True, False, 1)]


def _ids():
    return [f"{w.variant}-M{M}-{'c' if c else 'nc'}-{'tau' if t else 'notau'}-N{N}"
            for w, M, c, t, N in _cases()]


def _run(w, M, causal, tau, N, B=2, H=3):
    ws_ = w.replace(B=B, H=H, N=N, d=64, M=M, dtype="bf16")
    ins = workloads.make_inputs(ws_)
    t = workloads.draw_tau(ws_).astype(np.float64) if tau else None
    q, k = to_dev(ins["q"], "bf16"), to_dev(ins["k"], "bf16")
    W1, W2 = to_dev(ins["W1"], "f32"), to_dev(ins["W2"], "f32")
    tg = to_dev(t, "f32")
    shape = flexattn.shape_of(q, W1)
    ws = flexattn.awd_workspace(shape)
    n0 = flexattn.kernel_launches()
    loss = flexattn.awd_loss(q, k, W1, W2, causal, tau=tg, ws=ws)
    flexattn.check_status(ws)
    launches = flexattn.kernel_launches() - n0
    ref = oracle.awd(ins["q"], ins["k"], ins["W1"], ins["W2"], causal, tau=t)
    return loss, ref, launches, (q, k, W1, W2, tg, ws)


@pytest.mark.parametrize("w,M,causal,tau,N", _cases(), ids=_ids())
def test_awd_loss_matches_oracle(w, M, causal, tau, N):
    loss, ref, launches, _ = _run(w, M, causal, tau, N)
    assert launches == (5 if tau else 4)
    assert_close(to_host(loss), ref, "bf16", "awd loss")


def test_awd_nonpositive_kernel_estimates():
    """Large frequencies give negative kernel estimates (and some negative row sums); the
    loss still matches the oracle's reading (entries with R <= 0 count log 1e-6)."""
    w = WL[3].replace(B=1, H=2, N=200, d=64, M=64, dtype="bf16")
    ins = workloads.make_inputs(w)
    W1 = ins["W1"] * 6.0
    W2 = ins["W2"] * 6.0
    q, k = to_dev(ins["q"], "bf16"), to_dev(ins["k"], "bf16")
    loss = flexattn.awd_loss(q, k, to_dev(W1, "f32"), to_dev(W2, "f32"))
    torch.cuda.synchronize()
    ref = oracle.awd(ins["q"], ins["k"], W1, W2)
    assert_close(to_host(loss), ref, "bf16", "awd loss (negative estimates)")


def test_awd_repeatable():
    loss, _, _, (q, k, W1, W2, tg, ws) = _run(WL[2], 128, False, True, 300)
    again = flexattn.awd_loss(q, k, W1, W2, False, tau=tg, ws=ws)
    torch.cuda.synchronize()
    assert torch.equal(loss, again)
