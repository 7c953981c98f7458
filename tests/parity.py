"""Helpers shared by the GPU parity tests: device upload, tolerances, comparison."""
from __future__ import annotations

import numpy as np
import torch

# Tolerances stated for this path: fp32 storage, relative L2 <= 1e-4; bf16 storage with
# fp32 accumulation, relative L2 <= 2e-2 and max-abs <= 5e-2 (outputs and gradients).
F32_REL_L2 = 1e-4
BF16_REL_L2 = 2e-2
BF16_MAX_ABS = 5e-2


def to_dev(a, dtype):
    if a is None:
        return None
    t = torch.from_numpy(np.ascontiguousarray(a, dtype=np.float32)).cuda()
    return t.to(torch.bfloat16) if dtype == "bf16" else t


def to_host(t):
    return None if t is None else t.float().cpu().numpy().astype(np.float64)


def rel_l2(x, ref):
    return float(np.linalg.norm((x - ref).ravel()) / max(np.linalg.norm(ref.ravel()), 1e-300))


def max_abs(x, ref):
    return float(np.max(np.abs(x - ref)))


def assert_close(x, ref, dtype, what, max_abs_scale=1.0):
    """Compare a GPU result with the oracle under the tolerance of `dtype`.

    `max_abs_scale` states the magnitude the max-abs bound applies to (1 for O(1)
    outputs; the tensor's RMS for sums such as dW whose entries grow with B * N).
    """
    assert np.all(np.isfinite(x)), f"{what}: non-finite values"
    if np.linalg.norm(ref.ravel()) <= 1e-12 * np.sqrt(ref.size):
        # The exact result is zero (e.g. dq at a causal sequence of length 1, whose
        # output v_0 does not depend on q); relative error is undefined, so only the
        # absolute bound applies: fp32 rounding noise, or the stated bf16 max-abs bound.
        m = float(np.max(np.abs(x)))
        bound = 1e-5 if dtype == "f32" else BF16_MAX_ABS * max_abs_scale
        assert m <= bound, f"{what}: exact zero expected, max |x| = {m:.3e}"
        return 0.0
    r = rel_l2(x, ref)
    if dtype == "f32":
        assert r <= F32_REL_L2, f"{what}: rel L2 {r:.3e} > {F32_REL_L2}"
    else:
        m = max_abs(x, ref) / max_abs_scale
        assert r <= BF16_REL_L2, f"{what}: rel L2 {r:.3e} > {BF16_REL_L2}"
        assert m <= BF16_MAX_ABS, f"{what}: max-abs {m:.3e} > {BF16_MAX_ABS}"
    return r
