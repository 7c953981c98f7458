"""Gradient of the attention-weight distillation loss with respect to the kernel's
parameters (W1, W2, tau) on the GPU against the fp64 oracle: both variants, M = 64 and
128, causal and not, with and without the norm prefactor, sizes that leave a ragged last
block, a random upstream gradient per sequence; the full distillation workload in the
launch configuration the bench times, on a sample of its sequences (the upstream gradient
selects them); launch counts, the loss it returns, bit-exact repeatability; and, where
kernel estimates are negative (the gradient's pole at A = 0 makes it ill-conditioned
there), finite results and the loss."""
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


def _scale(ref):
    """dW and dtau are sums over B * N: the max-abs bound is relative to their RMS (an
    exactly zero gradient, N = 1, takes 1e-4: rounding of P / A against c / D only)."""
    rms = float(np.sqrt(np.mean(ref * ref)))
    return rms if rms > 1e-12 else 1e-4


def _compare(got, ref, what):
    for name, x, r in zip(("dW1", "dW2", "dtau"), got, ref):
        if r is None:
            assert x is None, f"{what}: {name} should be absent"
            continue
        assert_close(to_host(x), r, "bf16", f"{what} {name}", max_abs_scale=_scale(r))


def _inputs(w, tau):
    ins = workloads.make_inputs(w)
    t = workloads.draw_tau(w).astype(np.float64) if tau else None
    dev = dict(q=to_dev(ins["q"], "bf16"), k=to_dev(ins["k"], "bf16"),
               W1=to_dev(ins["W1"], "f32"), W2=to_dev(ins["W2"], "f32"), tau=to_dev(t, "f32"))
    return ins, t, dev


def _run(w, M, causal, tau, N, B=2, H=3, want_loss=True):
    ws_ = w.replace(B=B, H=H, N=N, d=64, M=M, dtype="bf16")
    ins, t, g = _inputs(ws_, tau)
    dl = np.random.default_rng(90 + N).uniform(0.5, 1.5, (B, H))
    ws = flexattn.awd_bwd_workspace(flexattn.shape_of(g["q"], g["W1"]))
    n0 = flexattn.kernel_launches()
    out = flexattn.awd_loss_bwd(g["q"], g["k"], g["W1"], g["W2"], causal, tau=g["tau"],
                                dloss=to_dev(dl, "f32"), ws=ws, want_loss=want_loss)
    flexattn.check_status(ws)
    launches = flexattn.kernel_launches() - n0
    ref = oracle.awd_bwd(ins["q"], ins["k"], ins["W1"], ins["W2"], causal, tau=t, dloss=dl)
    return out, ref, launches, (ins, t, g, dl, ws)


@pytest.mark.parametrize("w,M,causal,tau,N", _cases(), ids=_ids())
def test_awd_grad_matches_oracle(w, M, causal, tau, N):
    (loss, dW1, dW2, dtau), ref, launches, (ins, t, _, _, _) = _run(w, M, causal, tau, N)
    assert launches == (7 if tau else 6)
    _compare((dW1, dW2, dtau), ref, "awd grad")
    lref = oracle.awd(ins["q"], ins["k"], ins["W1"], ins["W2"], causal, tau=t)
    assert_close(to_host(loss), lref, "bf16", "awd loss (with the gradient)")


@pytest.mark.parametrize("tau", [False, True], ids=["notau", "tau"])
def test_awd_grad_full_workload_sampled(tau):
    """The full distillation workload (its grid and launch sequence); the upstream
    gradient is 1 on the sequences of batch entries 0 and 19 and 0 elsewhere, so the
    result is those sequences' gradient, which the oracle computes alone."""
    w = workloads.AWD
    ins, t, g = _inputs(w, tau)
    sample = [0, 19]
    dl = np.zeros((w.B, w.H), dtype=np.float32)
    dl[sample] = 1.0
    _, dW1, dW2, dtau = flexattn.awd_loss_bwd(g["q"], g["k"], g["W1"], g["W2"], w.causal,
                                              tau=g["tau"], dloss=to_dev(dl, "f32"))
    torch.cuda.synchronize()
    sub = workloads.make_inputs(w, bs=sample)
    ref = oracle.awd_bwd(sub["q"], sub["k"], sub["W1"], sub["W2"], w.causal, tau=t)
    _compare((dW1, dW2, dtau), ref, "awd grad, full workload")


def test_awd_grad_without_loss():
    """Without the loss output one reduction is skipped; the gradient is bit-identical."""
    a, _, la, _ = _run(WL[2], 128, True, True, 257)
    b, _, lb, _ = _run(WL[2], 128, True, True, 257, want_loss=False)
    assert (la, lb) == (7, 6) and b[0] is None
    for x, y in zip(a[1:], b[1:]):
        assert torch.equal(x, y)


def test_awd_grad_repeatable_and_loss_bit_exact():
    (loss, dW1, dW2, dtau), _, _, (_, _, g, dl, ws) = _run(WL[3], 64, False, True, 300)
    again = flexattn.awd_loss_bwd(g["q"], g["k"], g["W1"], g["W2"], False, tau=g["tau"],
                                  dloss=to_dev(dl, "f32"), ws=ws)
    only = flexattn.awd_loss(g["q"], g["k"], g["W1"], g["W2"], False, tau=g["tau"])
    torch.cuda.synchronize()
    for x, y in zip((loss, dW1, dW2, dtau), again):
        assert torch.equal(x, y)
    assert torch.equal(loss, only)


def test_awd_grad_nonpositive_estimates_finite():
    """Large frequencies: negative estimates and row sums.  The loss still matches the
    oracle; the gradient (pole at A = 0, so ill-conditioned here) is finite."""
    w = WL[3].replace(B=1, H=2, N=200, d=64, M=64, dtype="bf16")
    ins = workloads.make_inputs(w)
    W1, W2 = ins["W1"] * 6.0, ins["W2"] * 6.0
    q, k = to_dev(ins["q"], "bf16"), to_dev(ins["k"], "bf16")
    loss, dW1, dW2, _ = flexattn.awd_loss_bwd(q, k, to_dev(W1, "f32"), to_dev(W2, "f32"))
    torch.cuda.synchronize()
    assert_close(to_host(loss), oracle.awd(ins["q"], ins["k"], W1, W2), "bf16",
                 "awd loss (negative estimates)")
    assert torch.isfinite(dW1).all() and torch.isfinite(dW2).all()
