"""Recurrent decode step on the GPU against the fp64 oracle: single steps from a state
built by the oracle, and whole sequences stepped token by token against the oracle's
causal forward (every position) and its final running sums."""
import numpy as np
import pytest
import torch

import oracle
from paper_2606_27748_gb300 import flexattn, workloads
from parity import F32_REL_L2, assert_close, to_dev, to_host, rel_l2

pytestmark = pytest.mark.gpu

WL = workloads.ORDERED


@pytest.fixture(scope="module", autouse=True)
def library():
    assert torch.cuda.is_available(), "GPU tests need CUDA"
    from paper_2606_27748_gb300 import build
    build.build()
    flexattn.load()


def _cases():
    # (base workload, d, M, dtype)
    return [(WL[0], 32, 32, "f32"), (WL[1], 64, 64, "bf16"), (WL[2], 64, 128, "bf16"),
            (WL[3], 64, 64, "bf16"), (WL[2], 64, 128, "f32"), (WL[1], 128, 16, "f32")]


def _ids():
    return [f"{w.variant}-d{d}-M{M}-{dt}" for w, d, M, dt in _cases()]


def _inputs(w, B, H, N, d, M, dtype):
    ws_ = w.replace(B=B, H=H, N=N, d=d, M=M, dtype=dtype)
    return ws_, workloads.make_inputs(ws_)


@pytest.mark.parametrize("w,d,M,dtype", _cases(), ids=_ids())
def test_decode_steps_from_a_state(w, d, M, dtype):
    B, H, N = 2, 3, 20
    ws_, ins = _inputs(w, B, H, N, d, M, dtype)
    W1, W2 = ins["W1"], ins["W2"]
    S = np.zeros((B, H, 2 * M, d))
    z = np.zeros((B, H, 2 * M))
    for i in range(N - 3):  # state of the first N - 3 tokens, from the oracle
        _, _, S, z = oracle.decode(ins["q"][:, :, i], ins["k"][:, :, i], ins["v"][:, :, i],
                                   W1, W2, S, z)
    Sg = torch.from_numpy(S.astype(np.float32)).cuda()
    zg = torch.from_numpy(z.astype(np.float32)).cuda()
    for i in range(N - 3, N):
        q, k, v = (ins[n][:, :, i] for n in "qkv")
        ro, rd, S, z = oracle.decode(q, k, v, W1, W2, S, z)
        out, den = flexattn.linattn_decode(to_dev(q, dtype), to_dev(k, dtype), to_dev(v, dtype),
                                           to_dev(W1, "f32"), to_dev(W2, "f32"), Sg, zg)
        assert_close(to_host(out), ro, dtype, f"out step {i}")
        assert_close(to_host(den), rd, "f32", f"den step {i}")
        # the state is fp32 on both sides of the same (rounded) inputs
        assert rel_l2(to_host(Sg), S) <= F32_REL_L2 and rel_l2(to_host(zg), z) <= F32_REL_L2


@pytest.mark.parametrize("w,d,M,dtype", _cases(), ids=_ids())
def test_decode_sequence_equals_causal_forward(w, d, M, dtype):
    B, H, N = 2, 2, 150
    ws_, ins = _inputs(w, B, H, N, d, M, dtype)
    ro, rd = oracle.fwd(ins["q"], ins["k"], ins["v"], ins["W1"], ins["W2"], True)
    W1, W2 = to_dev(ins["W1"], "f32"), to_dev(ins["W2"], "f32")
    q, k, v = (to_dev(ins[n], dtype) for n in "qkv")
    S, z = flexattn.decode_state(B, H, M, d)
    outs, dens = [], []
    for i in range(N):
        o, dn = flexattn.linattn_decode(q[:, :, i].contiguous(), k[:, :, i].contiguous(),
                                        v[:, :, i].contiguous(), W1, W2, S, z)
        outs.append(to_host(o))
        dens.append(to_host(dn))
    assert_close(np.stack(outs, axis=2), ro, dtype, "decoded outputs")
    assert_close(np.stack(dens, axis=2), rd, "f32", "decoded den")
    # final running sums against the oracle's decode recurrence
    So = np.zeros((B, H, 2 * M, d))
    zo = np.zeros((B, H, 2 * M))
    for i in range(N):
        _, _, So, zo = oracle.decode(ins["q"][:, :, i], ins["k"][:, :, i], ins["v"][:, :, i],
                                     ins["W1"], ins["W2"], So, zo)
    assert rel_l2(to_host(S), So) <= F32_REL_L2 and rel_l2(to_host(z), zo) <= F32_REL_L2


def test_decode_launch_count():
    w = WL[2]
    ws_, ins = _inputs(w, 1, 2, 1, 64, 128, "bf16")
    S, z = flexattn.decode_state(1, 2, 128, 64)
    n0 = flexattn.kernel_launches()
    flexattn.linattn_decode(to_dev(ins["q"][:, :, 0], "bf16"), to_dev(ins["k"][:, :, 0], "bf16"),
                            to_dev(ins["v"][:, :, 0], "bf16"), to_dev(ins["W1"], "f32"),
                            to_dev(ins["W2"], "f32"), S, z)
    assert flexattn.kernel_launches() - n0 == 2  # features, then the state stream


def test_decode_reads_features_only_after_they_are_written():
    """The state kernel starts before the features kernel ends (its state copies overlap
    it) and must read phi only after the dependency wait.  Poison the workspace with NaN
    before every step: any early read shows up as a NaN, and the results must equal, bit
    for bit, those of a run whose workspace keeps the previous step's features."""
    w = WL[2]
    B, H, N, d, M = 64, 16, 24, 64, 128
    _, ins = _inputs(w, B, H, N, d, M, "bf16")
    W1, W2 = to_dev(ins["W1"], "f32"), to_dev(ins["W2"], "f32")
    q, k, v = (to_dev(ins[n], "bf16") for n in "qkv")
    toks = [tuple(t[:, :, i].contiguous() for t in (q, k, v)) for i in range(N)]
    runs = []
    for poison in (False, True):
        S, z = flexattn.decode_state(B, H, M, d)
        ws = flexattn.decode_workspace(B, H, M, d)
        outs = []
        for i in range(N):
            if poison:
                ws.view(torch.float32)[64:].fill_(float("nan"))  # past the 256-byte header
            o, dn = flexattn.linattn_decode(*toks[i], W1, W2, S, z, ws=ws)
            outs.append(torch.cat([o.float().flatten(), dn.flatten()]))
        torch.cuda.synchronize()
        runs.append((torch.stack(outs), S.clone(), z.clone()))
    (oa, Sa, za), (ob, Sb, zb) = runs
    assert torch.isfinite(ob).all() and torch.isfinite(Sb).all()
    assert torch.equal(oa, ob) and torch.equal(Sa, Sb) and torch.equal(za, zb)
