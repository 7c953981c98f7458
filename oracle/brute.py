"""Explicit N x N form of kernel attention, in numpy fp64.

TEST INFRASTRUCTURE ONLY (see the package docstring).  This module is written separately
from ``flex_oracle.c`` and with a different structure, so that the two can be checked
against each other:

  * the features of Flexformer_n are taken in the Monte Carlo sum form of Eq. (phi_non),
    (cos w_1i.x + cos w_2i.x, sin w_1i.x + sin w_2i.x) / (2 sqrt M), not in the
    product form that the C oracle uses;
  * attention is Eq. (attention) with sim(q_i, k_j) = phi(q_i) . phi(k_j) (Eq. kernel):
    the full N x N weight matrix is built, masked to j <= i when causal, and each row is
    divided by its sum -- no reassociation.
"""
from __future__ import annotations

import numpy as np


def features(x, W1, W2=None):
    """phi(x) for x [..., H, N, d] and frequencies [H, M, d] -> [..., H, N, 2M].

    Stationary: M^{-1/2} [cos(x W1^T), sin(x W1^T)]  (Eq. phi_n with sigma = 1).
    Nonstationary: (2 sqrt M)^{-1} [cos a + cos b, sin a + sin b], a = x W1^T, b = x W2^T.
    """
    x = np.asarray(x, dtype=np.float64)
    W1 = np.asarray(W1, dtype=np.float64)
    M = W1.shape[1]
    a = np.einsum("...hnd,hmd->...hnm", x, W1)
    if W2 is None:
        return np.concatenate([np.cos(a), np.sin(a)], axis=-1) / np.sqrt(M)
    b = np.einsum("...hnd,hmd->...hnm", x, np.asarray(W2, dtype=np.float64))
    return np.concatenate([np.cos(a) + np.cos(b), np.sin(a) + np.sin(b)], axis=-1) / (
        2.0 * np.sqrt(M))


def prefactored(x, W1, W2=None, tau=None):
    """phi~(x) = exp(|x|^2 / exp(tau)) phi(x) (Sec. 3.2), tau [H]; phi(x) if tau is None."""
    phi = features(x, W1, W2)
    if tau is None:
        return phi
    x = np.asarray(x, dtype=np.float64)
    t = np.asarray(tau, dtype=np.float64)[:, None]          # [H, 1] against [..., H, N]
    return np.exp(np.sum(x * x, axis=-1) / np.exp(t))[..., None] * phi


def kernel_matrix(q, k, W1, W2=None, tau=None):
    """K[..., i, j] = phi~(q_i) . phi~(k_j) (the prefactor on both sides, as printed)."""
    return np.einsum("...if,...jf->...ij", prefactored(q, W1, W2, tau),
                     prefactored(k, W1, W2, tau))


def attention(q, k, v, W1, W2=None, causal=True, tau=None):
    """(out, den): out_i = sum_j K_ij v_j / sum_j K_ij over j <= i (causal) or all j.
    With tau, den includes the query's prefactor (it is the literal row sum)."""
    K = kernel_matrix(q, k, W1, W2, tau)
    if causal:
        N = K.shape[-1]
        K = K * np.tril(np.ones((N, N)))
    den = K.sum(axis=-1)
    out = np.einsum("...ij,...je->...ie", K, np.asarray(v, dtype=np.float64)) / den[..., None]
    return out, den


def awd_loss(q, k, W1, W2=None, causal=False, tau=None, eps=1e-6):
    """Attention-weight distillation loss per sequence [..., H] with explicit N x N
    matrices: P = softmax(q k^T / sqrt(d)) (masked when causal), R = K~ / rowsum(K~) with
    the prefactored kernel K~ as printed (query and key factors), and
    L = -mean_i sum_j P_ij log R_ij; entries with R_ij <= 0 count log(eps)."""
    q = np.asarray(q, dtype=np.float64)
    k = np.asarray(k, dtype=np.float64)
    d = q.shape[-1]
    s = np.einsum("...id,...jd->...ij", q, k) / np.sqrt(d)
    K = kernel_matrix(q, k, W1, W2, tau)
    N = K.shape[-1]
    mask = np.tril(np.ones((N, N), dtype=bool)) if causal else np.ones((N, N), dtype=bool)
    s = np.where(mask, s, -np.inf)
    P = np.exp(s - s.max(axis=-1, keepdims=True))
    P = P / P.sum(axis=-1, keepdims=True)
    K = np.where(mask, K, 0.0)
    R = K / K.sum(axis=-1, keepdims=True)
    with np.errstate(divide="ignore", invalid="ignore"):
        logR = np.where(R > 0, np.log(np.where(R > 0, R, 1.0)), np.log(eps))
    return -np.sum(np.where(mask, P * logR, 0.0), axis=(-1, -2)) / N
