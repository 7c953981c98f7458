"""CUDA path against the fp64 oracle, element by element, on identical seeded inputs.

Reduced sizes span several chunks/tiles and a ragged tail; the full workload sizes run the
kernels in the bench's launch configuration and compare sampled whole sequences (all
batches of one head for dW, so the batch sum is exact).
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


def _gpu_fwd(w, ins, causal=None):
    causal = w.causal if causal is None else causal
    q, k, v = (to_dev(ins[n], w.dtype) for n in "qkv")
    W1, W2 = to_dev(ins["W1"], "f32"), to_dev(ins["W2"], "f32")
    shape = flexattn.shape_of(q, W1)
    ws = flexattn.workspace(shape, causal, False)
    out, den = flexattn.linattn_fwd(q, k, v, W1, W2, causal, ws=ws)
    flexattn.check_status(ws)
    return out, den


def _oracle_fwd(ins, causal):
    return oracle.fwd(ins["q"], ins["k"], ins["v"], ins["W1"], ins["W2"], causal)


def _small(w, N=1000):
    return w.replace(B=2, H=3, N=N)


@pytest.mark.parametrize("w", WL, ids=[w.name for w in WL])
def test_featmap(w):
    ws_ = _small(w, N=77)
    ins = workloads.make_inputs(ws_)
    for x in ("q", "k"):
        phi = flexattn.featmap(to_dev(ins[x], w.dtype), to_dev(ins["W1"], "f32"),
                               to_dev(ins["W2"], "f32"))
        torch.cuda.synchronize()
        ref = oracle.featmap(ins[x], ins["W1"], ins["W2"])
        assert_close(to_host(phi), ref, w.dtype, f"phi({x})")


@pytest.mark.parametrize("w", WL, ids=[w.name for w in WL])
@pytest.mark.parametrize("causal", [True, False])
def test_forward_reduced(w, causal):
    ws_ = _small(w)
    ins = workloads.make_inputs(ws_)
    out, den = _gpu_fwd(ws_, ins, causal)
    ro, rd = _oracle_fwd(ins, causal)
    assert_close(to_host(out), ro, w.dtype, "out")
    assert_close(to_host(den), rd, w.dtype, "den", max_abs_scale=float(np.abs(rd).max()))


@pytest.mark.parametrize("N", [1, 2, 3, 63, 64, 65, 127, 129, 300])
@pytest.mark.parametrize("w", [WL[1], WL[2]], ids=["stationary", "nonstationary"])
@pytest.mark.parametrize("causal", [True, False])
def test_forward_edges(w, N, causal):
    ws_ = w.replace(B=1, H=2, N=N)
    ins = workloads.make_inputs(ws_)
    out, _ = _gpu_fwd(ws_, ins, causal)
    ro, _ = _oracle_fwd(ins, causal)
    assert_close(to_host(out), ro, w.dtype, f"out N={N}")


def _gpu_bwd(w, ins, causal):
    q, k, v, dO = (to_dev(ins[n], w.dtype) for n in ("q", "k", "v", "dO"))
    W1, W2 = to_dev(ins["W1"], "f32"), to_dev(ins["W2"], "f32")
    out, den = _gpu_fwd(w, ins, causal)
    shape = flexattn.shape_of(q, W1)
    ws = flexattn.workspace(shape, causal, True)
    g = flexattn.linattn_bwd(q, k, v, W1, W2, causal, out, den, dO, ws=ws)
    flexattn.check_status(ws)
    return [to_host(t) for t in g]


def _compare_grads(w, g, r, what=""):
    names = ["dq", "dk", "dv", "dW1", "dW2"]
    for name, x, ref in zip(names, g, r):
        if ref is None:
            assert x is None
            continue
        scale = 1.0
        if name.startswith("dW"):  # sums over B * N: relative to their RMS (1 if zero)
            rms = float(np.sqrt(np.mean(ref * ref)))
            scale = rms if rms > 1e-12 else 1.0
        assert_close(x, ref, w.dtype, f"{what}{name}", max_abs_scale=scale)


@pytest.mark.parametrize("w", WL, ids=[w.name for w in WL])
@pytest.mark.parametrize("causal", [True, False])
def test_backward_reduced(w, causal):
    ws_ = _small(w, N=600).replace(backward=True)
    ins = workloads.make_inputs(ws_)
    g = _gpu_bwd(ws_, ins, causal)
    r = oracle.bwd(ins["q"], ins["k"], ins["v"], ins["W1"], ins["W2"], causal, ins["dO"])
    _compare_grads(w, g, r)


@pytest.mark.parametrize("N", [1, 2, 65, 129])
@pytest.mark.parametrize("causal", [True, False])
def test_backward_edges(N, causal):
    for w in (WL[1], WL[2]):
        ws_ = w.replace(B=2, H=1, N=N, backward=True)
        ins = workloads.make_inputs(ws_)
        g = _gpu_bwd(ws_, ins, causal)
        r = oracle.bwd(ins["q"], ins["k"], ins["v"], ins["W1"], ins["W2"], causal, ins["dO"])
        _compare_grads(w, g, r, f"N={N} ")


def _sampled(w, out_t, den_t, seqs):
    for (b, h) in seqs:
        ins = workloads.make_inputs(w, bs=[b], hs=[h])
        ro, rd = _oracle_fwd(ins, w.causal)
        assert_close(to_host(out_t[b:b + 1, h:h + 1]), ro, w.dtype, f"out[{b},{h}]")
        assert_close(to_host(den_t[b:b + 1, h:h + 1]), rd, w.dtype, f"den[{b},{h}]",
                     max_abs_scale=float(np.abs(rd).max()))


@pytest.mark.parametrize("w", WL, ids=[w.name for w in WL])
def test_forward_full_size_sampled(w):
    ins = workloads.make_inputs(w)
    out, den = _gpu_fwd(w, ins)
    del ins
    _sampled(w, out, den, [(0, 0), (w.B - 1, w.H - 1)])


def test_backward_full_size_head0():
    w = WL[4]
    ins = workloads.make_inputs(w)
    g = _gpu_bwd(w, ins, w.causal)
    del ins
    sub = workloads.make_inputs(w, hs=[0])
    r = oracle.bwd(sub["q"], sub["k"], sub["v"], sub["W1"], sub["W2"], w.causal, sub["dO"])
    g0 = [t[:, 0:1] for t in g[:3]] + [g[3][0:1], None]
    _compare_grads(w, g0, r)


def test_backward_full_size_noncausal_head0():
    """The non-causal backward on the long-sequence classification shape (8 x 8 x 65536,
    many chunk splits per sequence), sequences of head 0 against the oracle (dW of head 0
    sums the whole batch, so it is exact)."""
    w = WL[3].replace(backward=True)
    ins = workloads.make_inputs(w)
    g = _gpu_bwd(w, ins, w.causal)
    del ins
    sub = workloads.make_inputs(w, hs=[0])
    r = oracle.bwd(sub["q"], sub["k"], sub["v"], sub["W1"], sub["W2"], w.causal, sub["dO"])
    g0 = [t[:, 0:1] for t in g[:3]] + [g[3][0:1], g[4][0:1]]
    _compare_grads(w, g0, r)


@pytest.mark.parametrize("N", [700, 1800, 2000, 4097])
@pytest.mark.parametrize("w", [WL[1], WL[2]], ids=["stationary", "nonstationary"])
def test_forward_sequence_splits(w, N):
    """Few sequences and many chunks: the causal tensor-core path splits each sequence
    over 2 or 3 CTAs (k-only prefix pass + own segment); every position must match."""
    ws_ = w.replace(B=1, H=2, N=N)
    ins = workloads.make_inputs(ws_)
    out, den = _gpu_fwd(ws_, ins, True)
    ro, rd = _oracle_fwd(ins, True)
    assert_close(to_host(out), ro, w.dtype, f"out N={N}")
    assert_close(to_host(den), rd, w.dtype, "den", max_abs_scale=float(np.abs(rd).max()))


@pytest.mark.parametrize("w", [WL[1], WL[2]], ids=["stationary", "nonstationary"])
def test_dispatch_launch_counts_and_determinism(w):
    """The tensor-core entry points run (launch counts per call: causal forward 1, non-causal
    forward 3, causal backward 2, non-causal backward 4), and both backwards are bit-for-bit
    repeatable (dq, dk, dv are sums of at most two groups, each added by the CTA that owns
    the row; the non-causal totals and dW are reduced in a fixed order)."""
    ws_ = w.replace(B=2, H=2, N=700, backward=True)
    ins = workloads.make_inputs(ws_)
    n0 = flexattn.kernel_launches()
    _gpu_fwd(ws_, ins, True)
    assert flexattn.kernel_launches() - n0 == 1
    n0 = flexattn.kernel_launches()
    _gpu_fwd(ws_, ins, False)
    assert flexattn.kernel_launches() - n0 == 3
    n0 = flexattn.kernel_launches()
    g1 = _gpu_bwd(ws_, ins, True)
    assert flexattn.kernel_launches() - n0 == 1 + 2  # the forward it runs first + backward
    g2 = _gpu_bwd(ws_, ins, True)
    n0 = flexattn.kernel_launches()
    h1 = _gpu_bwd(ws_, ins, False)
    assert flexattn.kernel_launches() - n0 == 3 + 4  # the non-causal forward + backward
    h2 = _gpu_bwd(ws_, ins, False)
    for a, b in list(zip(g1, g2)) + list(zip(h1, h2)):
        if a is None:
            assert b is None
        else:
            assert np.array_equal(a, b)
