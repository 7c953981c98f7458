"""Seeded synthetic workloads shared by the tests, the smoke check and the bench.

This module only draws random inputs and rounds them to the storage type; it holds none
of the attention arithmetic.  Both the CUDA path and the CPU oracle consume what it
returns, so the two always see bit-identical inputs.

The five workloads stand in for the paper's language-modelling (head size 64, 8-16 heads,
n = 64 frequencies; Appendix Table "wiki params", Sec. 4.2) and long-sequence
classification (LRA, N = 1K-4K, d = 64; Sec. 4.1) settings, extended to longer N.

Draw recipe: every (tensor, b, h) slice has its own PCG64 stream, seeded by
``(seed, tensor_id, b, h)`` (frequencies: ``(seed, tensor_id, h)``), so any subset of
sequences can be regenerated without drawing the rest.  Tensor ids follow the draw order
q=0, k=1, v=2, W1=3, W2=4, dO=5 (6: the q/k offset of large-argument inputs).  Values are
drawn in float32; bf16 workloads are then rounded once to bf16 (round to nearest even) and
the rounded values are what both sides use.
"""
from __future__ import annotations

import dataclasses

import numpy as np

Q, K, V, W1, W2, DO, OFFSET = range(7)


@dataclasses.dataclass(frozen=True)
class Workload:
    name: str
    variant: str          # "s": stationary (W1 only); "n": nonstationary (W1, W2)
    causal: bool
    dtype: str            # "f32" or "bf16" storage of q, k, v, out, dq, dk, dv
    B: int
    H: int
    N: int
    d: int
    M: int                # frequencies per set; feature dimension d' = 2M
    qk_scale: float       # q, k ~ N(0, 1) * qk_scale
    v_dist: str           # "normal": N(0, 1); "uniform": U(-1, 1)
    seed: int
    backward: bool = False
    decode: bool = False  # recurrent decode steps: one new token per sequence per step
    awd: bool = False     # attention-weight distillation loss (q, k only)
    # Large projection arguments |x . w| (the regime of trained frequencies): q and k of
    # head h share an offset vector m_h ~ N(0, qk_offset^2 I) (every batch entry), and the
    # frequencies are drawn with standard deviation w_scale / sqrt(d).
    qk_offset: float = 0.0
    w_scale: float = 1.0

    @property
    def tokens(self) -> int:
        return self.B * self.N

    @property
    def token_heads(self) -> int:
        return self.B * self.H * self.N

    def replace(self, **kw) -> "Workload":
        return dataclasses.replace(self, **kw)


WORKLOADS = {
    w.name: w for w in [
        Workload("s_noncausal_f32_B1H1N256_d32M32", "s", False, "f32", 1, 1, 256, 32, 32,
                 1.0, "normal", 0),
        Workload("s_causal_bf16_B8H12N4096_d64M64", "s", True, "bf16", 8, 12, 4096, 64, 64,
                 64 ** -0.25, "normal", 2),
        Workload("n_causal_bf16_B4H16N16384_d64M128", "n", True, "bf16", 4, 16, 16384, 64,
                 128, 64 ** -0.25, "normal", 3),
        Workload("n_noncausal_bf16_B8H8N65536_d64M64", "n", False, "bf16", 8, 8, 65536, 64,
                 64, 64 ** -0.25, "uniform", 4),
        Workload("s_causal_train_bf16_B8H12N8192_d64M128", "s", True, "bf16", 8, 12, 8192, 64,
                 128, 64 ** -0.25, "normal", 5, backward=True),
    ]
}
ORDERED = list(WORKLOADS.values())  # the five configurations
HEADLINE = ORDERED[2]
# Serving shape for the recurrent decode step: 256 sequences x 16 heads, the headline's
# per-head sizes; the fp32 running state (268 MB) exceeds L2, so every step streams it.
# N = tokens cycled through by the bench.
DECODE = Workload("n_decode_bf16_B256H16_d64M128", "n", True, "bf16", 256, 16, 64, 64, 128,
                  64 ** -0.25, "normal", 6, decode=True)
WORKLOADS[DECODE.name] = DECODE
# The distillation setting: a 125M RoBERTa encoder (8 heads, head size 64) converted with
# n = d = 64 frequencies, batch 32, sequences of 512 tokens (non-causal).
AWD = Workload("n_awd_bf16_B32H8N512_d64M64", "n", False, "bf16", 32, 8, 512, 64, 64,
               64 ** -0.25, "normal", 7, awd=True)
WORKLOADS[AWD.name] = AWD
# A training step (forward + backward) on the long-sequence classification shape: the
# non-causal backward.
NONCAUSAL_TRAIN = ORDERED[3].replace(name="n_noncausal_train_bf16_B8H8N65536_d64M64",
                                     backward=True)
WORKLOADS[NONCAUSAL_TRAIN.name] = NONCAUSAL_TRAIN
# One distillation training step on the same batch: the loss and its gradient with respect
# to the kernel's parameters (W1, W2; tau with the prefactor).
AWD_TRAIN = AWD.replace(name="n_awd_train_bf16_B32H8N512_d64M64", backward=True)
WORKLOADS[AWD_TRAIN.name] = AWD_TRAIN


def bf16_bits(x: np.ndarray) -> np.ndarray:
    """float32 -> bf16 bit patterns (uint16), round to nearest even.  Inputs are finite."""
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32)
    r = (u + np.uint32(0x7FFF) + ((u >> np.uint32(16)) & np.uint32(1))) >> np.uint32(16)
    return r.astype(np.uint16)


def bf16_to_f32(bits: np.ndarray) -> np.ndarray:
    return (bits.astype(np.uint32) << np.uint32(16)).view(np.float32)


def _stream(*key):
    return np.random.Generator(np.random.PCG64(list(key)))


def _draw_seq(w: Workload, tensor: int, b: int, h: int, N: int) -> np.ndarray:
    g = _stream(w.seed, tensor, b, h)
    if tensor in (Q, K):
        x = g.standard_normal((N, w.d), dtype=np.float32) * np.float32(w.qk_scale)
        if w.qk_offset:
            x += draw_offset(w, [h])[0]
        return x
    if tensor == V and w.v_dist == "uniform":
        return g.uniform(-1.0, 1.0, (N, w.d)).astype(np.float32)
    return g.standard_normal((N, w.d), dtype=np.float32)


def draw_offset(w: Workload, hs=None) -> np.ndarray:
    """float32 [len(hs), d]: the offset m_h shared by q and k of head h (zeros if none)."""
    hs = range(w.H) if hs is None else hs
    out = np.zeros((len(hs), w.d), dtype=np.float32)
    if w.qk_offset:
        for j, h in enumerate(hs):
            out[j] = _stream(w.seed, OFFSET, h).standard_normal(w.d, dtype=np.float32)
        out *= np.float32(w.qk_offset)
    return out


def draw_activation(w: Workload, tensor: int, bs=None, hs=None, N=None) -> np.ndarray:
    """float32 [len(bs), len(hs), N, d] for q, k, v or dO, rounded to bf16 if w.dtype is."""
    bs = range(w.B) if bs is None else bs
    hs = range(w.H) if hs is None else hs
    N = w.N if N is None else N
    out = np.empty((len(bs), len(hs), N, w.d), dtype=np.float32)
    for i, b in enumerate(bs):
        for j, h in enumerate(hs):
            out[i, j] = _draw_seq(w, tensor, b, h, N)
    if w.dtype == "bf16":
        out = bf16_to_f32(bf16_bits(out))
    return out


def draw_frequencies(w: Workload, tensor: int, hs=None) -> np.ndarray:
    """float32 [len(hs), M, d] with entries ~ N(0, w_scale^2 / d)."""
    hs = range(w.H) if hs is None else hs
    out = np.empty((len(hs), w.M, w.d), dtype=np.float32)
    for j, h in enumerate(hs):
        out[j] = _stream(w.seed, tensor, h).standard_normal((w.M, w.d), dtype=np.float32)
    return out * np.float32(w.w_scale / np.sqrt(w.d))


def draw_tau(w: Workload, hs=None) -> np.ndarray:
    """Per-head tau of the norm prefactor exp(|x|^2 / exp(tau)): ln(2 sqrt d) (the fixed
    softmax-kernel value the learnable exp(tau) replaces) plus -0.25, 0, +0.25 by head.
    With q, k ~ N(0, 1) d^-1/4 the key weights spread over about 1.3-2.1."""
    heads = range(w.H) if hs is None else hs
    return np.array([np.log(2.0 * np.sqrt(w.d)) + 0.25 * ((h % 3) - 1) for h in heads],
                    dtype=np.float32)


def make_inputs(w: Workload, bs=None, hs=None, N=None) -> dict:
    """All inputs of one workload (or of a subset of its sequences) as float32 arrays.

    Keys: q, k, v, W1, W2 (None for the stationary variant), dO (None unless backward).
    """
    ins = {
        "q": draw_activation(w, Q, bs, hs, N),
        "k": draw_activation(w, K, bs, hs, N),
        "v": draw_activation(w, V, bs, hs, N),
        "W1": draw_frequencies(w, W1, hs),
        "W2": draw_frequencies(w, W2, hs) if w.variant == "n" else None,
        "dO": draw_activation(w, DO, bs, hs, N) if w.backward else None,
    }
    return ins
