"""The norm prefactor exp(|x|^2 / exp(tau)) of Sec. 3.2 on the GPU against the fp64
oracle: forward (out, den), backward (dq, dk, dv, dW1, dW2, dtau) and decode steps, both
variants, causal and non-causal, bf16 and fp32 storage, at sizes that span several chunks
and a ragged tail."""
import numpy as np
import pytest
import torch

import oracle
from paper_2606_27748_gb300 import flexattn, workloads
from parity import BF16_REL_L2, F32_REL_L2, assert_close, rel_l2, to_dev, to_host

pytestmark = pytest.mark.gpu

WL = workloads.ORDERED


@pytest.fixture(scope="module", autouse=True)
def library():
    assert torch.cuda.is_available(), "GPU tests need CUDA"
    from paper_2606_27748_gb300 import build
    build.build()
    flexattn.load()


def _cases():
    # (base workload, causal, d, M, dtype): both variants, both masks, both storage types
    return [(WL[0], False, 32, 32, "f32"), (WL[1], True, 64, 64, "bf16"),
            (WL[2], True, 64, 128, "bf16"), (WL[3], False, 64, 64, "bf16"),
            (WL[2], True, 64, 32, "f32"), (WL[1], False, 64, 64, "bf16")]


def _ids():
    return [f"{w.variant}-{'c' if c else 'nc'}-d{d}-M{M}-{dt}" for w, c, d, M, dt in _cases()]


def _setup(w, causal, d, M, dtype, B=2, H=3, N=300):
    ws_ = w.replace(B=B, H=H, N=N, d=d, M=M, dtype=dtype, causal=causal, backward=True)
    ins = workloads.make_inputs(ws_)
    ins["tau"] = workloads.draw_tau(ws_).astype(np.float64)
    return ws_, ins


def _dev(ins, dtype):
    q, k, v, dO = (to_dev(ins[n], dtype) for n in ("q", "k", "v", "dO"))
    return q, k, v, dO, to_dev(ins["W1"], "f32"), to_dev(ins["W2"], "f32"), to_dev(ins["tau"], "f32")


@pytest.mark.parametrize("w,causal,d,M,dtype", _cases(), ids=_ids())
def test_forward_with_prefactor(w, causal, d, M, dtype):
    _, ins = _setup(w, causal, d, M, dtype)
    q, k, v, _, W1, W2, tau = _dev(ins, dtype)
    out, den = flexattn.linattn_fwd(q, k, v, W1, W2, causal, tau=tau)
    ro, rd = oracle.fwd(ins["q"], ins["k"], ins["v"], ins["W1"], ins["W2"], causal,
                        tau=ins["tau"])
    assert_close(to_host(out), ro, dtype, "out")
    assert rel_l2(to_host(den), rd) <= (F32_REL_L2 if dtype == "f32" else 1e-2), "den"
    # the prefactor changes the result: the weights are not all equal
    r0, _ = oracle.fwd(ins["q"], ins["k"], ins["v"], ins["W1"], ins["W2"], causal)
    assert rel_l2(r0, ro) > 1e-3


@pytest.mark.parametrize("w,causal,d,M,dtype", _cases(), ids=_ids())
def test_backward_with_prefactor(w, causal, d, M, dtype):
    _, ins = _setup(w, causal, d, M, dtype)
    q, k, v, dO, W1, W2, tau = _dev(ins, dtype)
    out, den = flexattn.linattn_fwd(q, k, v, W1, W2, causal, tau=tau)
    g = flexattn.linattn_bwd(q, k, v, W1, W2, causal, out, den, dO, tau=tau)
    torch.cuda.synchronize()
    r = oracle.bwd(ins["q"], ins["k"], ins["v"], ins["W1"], ins["W2"], causal, ins["dO"],
                   tau=ins["tau"])
    for name, x, ref in zip(("dq", "dk", "dv", "dW1", "dW2"), g, r):
        if ref is None:
            assert x is None
            continue
        scale = 1.0 if name in ("dq", "dk", "dv") else float(np.sqrt(np.mean(ref * ref)))
        assert_close(to_host(x), ref, dtype, name, max_abs_scale=scale)
    # dtau is the remainder of a sum over every key that cancels exactly when the key norms
    # are equal; the kernels subtract that common part exactly (the s_j of a sequence sum to
    # zero), so dtau keeps the stated tolerances.
    err = rel_l2(to_host(g[5]), r[5])
    assert err <= (F32_REL_L2 if dtype == "f32" else BF16_REL_L2), f"dtau: rel L2 {err:.3e}"


@pytest.mark.parametrize("w,causal,d,M,dtype", [c for c in _cases() if c[1]],
                         ids=[i for i, c in zip(_ids(), _cases()) if c[1]])
def test_decode_with_prefactor(w, causal, d, M, dtype):
    """Stepping a sequence through the decode entry point with tau reproduces every row of
    the oracle's causal forward with tau, and ends in its running sums."""
    B, H, N = 2, 3, 40
    _, ins = _setup(w, True, d, M, dtype, B=B, H=H, N=N)
    q, k, v, _, W1, W2, tau = _dev(ins, dtype)
    ro, rd = oracle.fwd(ins["q"], ins["k"], ins["v"], ins["W1"], ins["W2"], True,
                        tau=ins["tau"])
    S, z = flexattn.decode_state(B, H, M, d)
    ws = flexattn.decode_workspace(B, H, M, d)
    outs, dens = [], []
    for i in range(N):
        o, dn = flexattn.linattn_decode(q[:, :, i].contiguous(), k[:, :, i].contiguous(),
                                        v[:, :, i].contiguous(), W1, W2, S, z, ws=ws, tau=tau)
        outs.append(to_host(o))
        dens.append(to_host(dn))
    assert_close(np.stack(outs, axis=2), ro, dtype, "decoded outputs")
    assert rel_l2(np.stack(dens, axis=2), rd) <= F32_REL_L2, "decoded den"
    So = np.zeros((B, H, 2 * M, d))
    zo = np.zeros((B, H, 2 * M))
    for i in range(N):
        _, _, So, zo = oracle.decode(ins["q"][:, :, i], ins["k"][:, :, i], ins["v"][:, :, i],
                                     ins["W1"], ins["W2"], So, zo, tau=ins["tau"])
    assert rel_l2(to_host(S), So) <= F32_REL_L2 and rel_l2(to_host(z), zo) <= F32_REL_L2


@pytest.mark.parametrize("causal,launches", [(True, 2), (False, 4)])
def test_tensor_core_forward_takes_the_prefactor(causal, launches):
    """bf16 d = 64 shapes keep the tensor-core forward with tau: one pass over k for the
    key weights, then the usual kernels (causal 1, non-causal 3)."""
    w = WL[2] if causal else WL[3]
    _, ins = _setup(w, causal, 64, 64, "bf16", N=700)
    q, k, v, _, W1, W2, tau = _dev(ins, "bf16")
    shape = flexattn.shape_of(q, W1)
    ws = flexattn.workspace(shape, causal, False)
    n0 = flexattn.kernel_launches()
    out, den = flexattn.linattn_fwd(q, k, v, W1, W2, causal, ws=ws, tau=tau)
    flexattn.check_status(ws)
    assert flexattn.kernel_launches() - n0 == launches
    ro, _ = oracle.fwd(ins["q"], ins["k"], ins["v"], ins["W1"], ins["W2"], causal,
                       tau=ins["tau"])
    assert_close(to_host(out), ro, "bf16", "out")


@pytest.mark.parametrize("causal,launches", [(True, 3), (False, 5)], ids=["causal", "non-causal"])
@pytest.mark.parametrize("w,M", [(WL[2], 128), (WL[1], 64)], ids=["n-M128", "s-M64"])
def test_tensor_core_backward_takes_the_prefactor(w, M, causal, launches):
    """bf16 d = 64 keeps the tensor-core backward with tau: the key-weight pass, then causal:
    the two-scan kernel (bf16 dq, dk, dv written directly) and the dW/dtau reduction;
    non-causal: the partial states, their totals, the gradient kernel and the reduction.
    The result matches the oracle and repeats bit for bit."""
    _, ins = _setup(w, causal, 64, M, "bf16", N=520)
    q, k, v, dO, W1, W2, tau = _dev(ins, "bf16")
    out, den = flexattn.linattn_fwd(q, k, v, W1, W2, causal, tau=tau)
    shape = flexattn.shape_of(q, W1)
    ws = flexattn.workspace(shape, causal, True)
    runs = []
    for _ in range(2):
        n0 = flexattn.kernel_launches()
        g = flexattn.linattn_bwd(q, k, v, W1, W2, causal, out, den, dO, ws=ws, tau=tau)
        flexattn.check_status(ws)
        assert flexattn.kernel_launches() - n0 == launches
        runs.append([None if x is None else x.clone() for x in g])
    for a, b in zip(*runs):
        assert (a is None and b is None) or torch.equal(a, b), "not bit-exact repeatable"
    r = oracle.bwd(ins["q"], ins["k"], ins["v"], ins["W1"], ins["W2"], causal, ins["dO"],
                   tau=ins["tau"])
    g = runs[0]
    for name, x, ref in zip(("dq", "dk", "dv", "dW1", "dW2"), g, r):
        if ref is None:
            continue
        scale = 1.0 if name in ("dq", "dk", "dv") else float(np.sqrt(np.mean(ref * ref)))
        assert_close(to_host(x), ref, "bf16", name, max_abs_scale=scale)
    err = rel_l2(to_host(g[5]), r[5])
    assert err <= BF16_REL_L2, f"dtau: rel L2 {err:.3e}"
