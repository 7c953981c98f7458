"""Helpers shared by the GPU parity tests: device upload, tolerances, comparison."""
from __future__ import annotations

import numpy as np
import torch

# Tolerances stated for this path: fp32 storage, relative L2 <= 1e-4; bf16 storage with
# fp32 accumulation, relative L2 <= 2e-2 and max-abs <= 5e-2 (outputs and gradients).
F32_REL_L2 = 1e-4
BF16_REL_L2 = 2e-2
BF16_MAX_ABS = 5e-2
ZERO_ABS = 1e-5  # an exactly-zero result


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
        # The exact result is zero (e.g. dq, dk and dW at a sequence of length 1, whose
        # output v_0 depends on neither q, k nor W); relative error is undefined.  The
        # kernels form the two cancelling terms from the same rounded operands (g and
        # c = -(g . out) from the bf16 g that feeds the MMAs), so the zero comes out to
        # fp32 rounding for either storage type.
        m = float(np.max(np.abs(x)))
        assert m <= ZERO_ABS, f"{what}: exact zero expected, max |x| = {m:.3e}"
        return 0.0
    r = rel_l2(x, ref)
    if dtype == "f32":
        assert r <= F32_REL_L2, f"{what}: rel L2 {r:.3e} > {F32_REL_L2}"
    else:
        m = max_abs(x, ref) / max_abs_scale
        assert r <= BF16_REL_L2, f"{what}: rel L2 {r:.3e} > {BF16_REL_L2}"
        assert m <= BF16_MAX_ABS, f"{what}: max-abs {m:.3e} > {BF16_MAX_ABS}"
    return r


def assert_close_offset_split(x, ref, x0_rms, offsets, dtype, what):
    """dW1/dW2 [H, M, d] of inputs whose q and k of head h share a large offset m_h.

    dW_h = sum_t da_t x_t^T with x_t = m_h + x0_t.  Its component along m_h,
    (sum_t da_t) |m_h|, is a sum whose terms cancel (exactly, for the stationary kernel:
    phi_s(q + m) . phi_s(k + m) = phi_s(q) . phi_s(k)), so with bf16 operands its error
    grows with the condition number kappa = |m_h| / rms |x0_t| of that sum, not with the
    result.  The component orthogonal to m_h is held to the stated bound; the component
    along m_h to the stated relative bound times kappa.
    """
    scale = float(np.sqrt(np.mean(ref * ref)))
    mh = offsets / np.linalg.norm(offsets, axis=1, keepdims=True)  # [H, d]
    err = x - ref
    along = np.einsum("hfd,hd->hf", err, mh)
    perp = err - along[..., None] * mh[:, None, :]
    rn = float(np.linalg.norm(ref))
    kappa = float(np.linalg.norm(offsets, axis=1).max() / x0_rms)
    tol = F32_REL_L2 if dtype == "f32" else BF16_REL_L2
    r_perp = float(np.linalg.norm(perp)) / rn
    r_along = float(np.linalg.norm(along)) / rn
    assert np.all(np.isfinite(x)), f"{what}: non-finite values"
    assert r_perp <= tol, f"{what}: orthogonal part rel L2 {r_perp:.3e} > {tol}"
    if dtype != "f32":
        m = float(np.abs(perp).max()) / scale
        assert m <= BF16_MAX_ABS, f"{what}: orthogonal part max-abs {m:.3e} > {BF16_MAX_ABS}"
    assert r_along <= tol * kappa, (
        f"{what}: part along the offset rel L2 {r_along:.3e} > {tol} x kappa {kappa:.1f}")
    return r_perp, r_along, kappa
