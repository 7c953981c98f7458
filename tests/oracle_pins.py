"""Checks that pin the fp64 oracle to facts fixed by the paper and by mathematics.

Each ``pin_*`` function takes one compiled copy of the C oracle (``oracle.Oracle``) and
raises AssertionError when the copy disagrees with the fact it checks.  The same
functions run against the real oracle (all must pass) and against copies with planted
mistakes (at least one must fail), so every pin is itself checked.

Facts used (none is the oracle's own formula retyped):
  * x = 0 gives phi = M^{-1/2} [1..1, 0..0]: fixes feature order (cos block first,
    Eq. phi_n) and the scale.
  * |phi_s(x)| = 1 (cos^2 + sin^2 = 1): fixes the stationary scale.
  * Eq. (phi_non): the product form equals the Monte Carlo sum form (sum-to-product).
  * W2 = W1 reduces Flexformer_n to Flexformer_s.
  * Bochner (Thm. bochner): with w ~ N(0, s^-2 I), phi(x).phi(y) -> exp(-|x-y|^2 / 2 s^2).
  * Yaglom (Thm. yaglom) with independent Gaussian W1, W2:
      E = 1/2 exp(-|x-y|^2 / 2 s^2) + 1/2 exp(-(|x|^2 + |y|^2) / 2 s^2).
  * Eq. (linear att) is an exact reassociation of Eq. (attention): the C linear form
    equals the numpy N x N form (different module, different feature form); so does the
    C decode recurrence run token by token, and its state equals the numpy running sums.
  * d = 1, M = 1: phi_s(q).phi_s(k) = cos(w (q - k)) in closed form.
  * causal output at the last position equals the non-causal output.
  * causal O_0 = v_0; constant v = c gives O = c (rows of weights sum to one).
  * gradients: central finite differences of the numpy N x N form; the exact invariants
    sum_j dv_j = sum_i dO_i, translation invariance of the stationary kernel
    (sum dq + sum dk = 0) and Euler's identity for a = W x
    (<dW1, W1> + <dW2, W2> = sum <dq, q> + sum <dk, k>).
  * the norm prefactor exp(|x|^2 / exp(tau)) (Sec. 3.2): the linear form with the key
    weight equals the N x N form with the factor on queries and keys as printed; it
    vanishes as tau grows; keys of equal norm make it a common factor (O unchanged);
    finite differences (dq, dk, dv, dW, dtau); the scaling identity
    <dW, W> = sum <dq, q> + <dk, k> + 2 dtau (x -> l x, W -> W / l, tau -> tau + 2 ln l).
  * the distillation loss: the C loss equals the explicit-matrix numpy form; one key gives
    0; d = 1, M = 1 in closed form (cos kernel, softmax teacher); Gibbs' inequality
    (loss >= the teacher's entropy); keys of equal norm make tau irrelevant; entries with
    a non-positive normalised weight count log 1e-6 in both forms.
  * its gradient with respect to W1, W2 and tau: central finite differences of the numpy
    form (cases with negative kernel entries); d = 1, M = 1 in closed form; one key gives
    0; keys of equal norm give dtau = 0; W2 = W1 gives dW1 + dW2 = the stationary
    gradient.
"""
from __future__ import annotations

import numpy as np

from oracle import brute


def _rng(seed):
    return np.random.default_rng(seed)


def _case(seed, B, H, N, d, M, variant, qk_scale=0.5):
    g = _rng(seed)
    q = g.standard_normal((B, H, N, d)) * qk_scale
    k = g.standard_normal((B, H, N, d)) * qk_scale
    v = g.standard_normal((B, H, N, d))
    W1 = g.standard_normal((H, M, d)) / np.sqrt(d)
    W2 = g.standard_normal((H, M, d)) / np.sqrt(d) if variant == "n" else None
    return q, k, v, W1, W2


def _rel(a, b):
    return float(np.max(np.abs(a - b)) / max(np.max(np.abs(b)), 1e-300))


def pin_origin_features(orc):
    for W2 in (None, np.full((2, 5, 3), 0.3)):
        W1 = _rng(1).standard_normal((2, 5, 3))
        phi = orc.featmap(np.zeros((1, 2, 4, 3)), W1, W2)
        expect = np.concatenate([np.ones(5), np.zeros(5)]) / np.sqrt(5)
        assert np.allclose(phi, expect, rtol=0, atol=1e-15), "phi(0) order or scale"


def pin_stationary_unit_norm(orc):
    q, _, _, W1, _ = _case(2, 2, 3, 7, 5, 11, "s", qk_scale=3.0)
    phi = orc.featmap(q, W1)
    assert np.allclose(np.sum(phi * phi, axis=-1), 1.0, rtol=0, atol=1e-13), "|phi_s| != 1"


def pin_sum_to_product(orc):
    q, _, _, W1, W2 = _case(3, 2, 2, 9, 6, 13, "n", qk_scale=2.0)
    prod = orc.featmap(q, W1, W2)
    assert _rel(prod, brute.features(q, W1, W2)) < 1e-13, "product form != sum form (numpy)"
    assert _rel(prod, orc.featmap_sumform(q, W1, W2)) < 1e-13, "product form != sum form (C)"


def pin_w2_equals_w1(orc):
    q, _, _, W1, _ = _case(4, 1, 2, 6, 4, 8, "s", qk_scale=2.0)
    assert _rel(orc.featmap(q, W1, W1.copy()), orc.featmap(q, W1)) < 1e-15, "W2=W1 != phi_s"


def _kernel_estimate(orc, x, y, W1, W2):
    """phi(x).phi(y) and the per-frequency terms whose mean it is."""
    px = orc.featmap(x[None, None, None], W1[None], None if W2 is None else W2[None])[0, 0, 0]
    py = orc.featmap(y[None, None, None], W1[None], None if W2 is None else W2[None])[0, 0, 0]
    M = W1.shape[0]
    terms = M * (px[:M] * py[:M] + px[M:] * py[M:])
    return float(px @ py), terms


def pin_bochner(orc):
    g = _rng(5)
    d, M, sigma = 6, 1 << 16, 1.3
    W = g.standard_normal((M, d)) / sigma
    for _ in range(3):
        x, y = g.standard_normal(d) * 0.8, g.standard_normal(d) * 0.8
        est, terms = _kernel_estimate(orc, x, y, W, None)
        exact = np.exp(-np.sum((x - y) ** 2) / (2 * sigma ** 2))
        assert abs(est - exact) <= 5 * terms.std() / np.sqrt(M), "Bochner estimate off"


def pin_yaglom(orc):
    g = _rng(6)
    d, M, sigma = 6, 1 << 16, 1.3
    W1 = g.standard_normal((M, d)) / sigma
    W2 = g.standard_normal((M, d)) / sigma
    for _ in range(3):
        x, y = g.standard_normal(d) * 0.8, g.standard_normal(d) * 0.8
        est, terms = _kernel_estimate(orc, x, y, W1, W2)
        exact = 0.5 * np.exp(-np.sum((x - y) ** 2) / (2 * sigma ** 2)) + 0.5 * np.exp(
            -(np.sum(x * x) + np.sum(y * y)) / (2 * sigma ** 2))
        assert abs(est - exact) <= 5 * terms.std() / np.sqrt(M), "Yaglom estimate off"


def pin_linear_equals_brute(orc):
    for variant in ("s", "n"):
        for causal in (True, False):
            for N in (1, 2, 3, 17, 64, 256):
                q, k, v, W1, W2 = _case(10 + N, 2, 2, N, 5, 7, variant)
                out, den = orc.fwd(q, k, v, W1, W2, causal)
                bo, bd = brute.attention(q, k, v, W1, W2, causal)
                assert _rel(den, bd) < 1e-12, f"den {variant} causal={causal} N={N}"
                assert _rel(out, bo) < 1e-11, f"out {variant} causal={causal} N={N}"


def pin_decode_equals_brute(orc):
    """Token-by-token decode from the zero state reproduces every row of the causal N x N
    form, and the state it carries is sum_j phi(k_j) v_j^T, sum_j phi(k_j) with the numpy
    features (sum form for n)."""
    for variant in ("s", "n"):
        B, H, N, d, M = 2, 2, 9, 5, 7
        q, k, v, W1, W2 = _case(40, B, H, N, d, M, variant)
        bo, bd = brute.attention(q, k, v, W1, W2, True)
        S = np.zeros((B, H, 2 * M, d))
        z = np.zeros((B, H, 2 * M))
        for i in range(N):
            out, den, S, z = orc.decode(q[:, :, i], k[:, :, i], v[:, :, i], W1, W2, S, z)
            assert _rel(den, bd[:, :, i]) < 1e-12, f"decode den {variant} i={i}"
            assert _rel(out, bo[:, :, i]) < 1e-11, f"decode out {variant} i={i}"
        pk = brute.features(k, W1, W2)
        assert _rel(S, np.einsum("bhnf,bhne->bhfe", pk, v)) < 1e-12, f"decode S {variant}"
        assert _rel(z, pk.sum(axis=2)) < 1e-12, f"decode z {variant}"


def pin_closed_form_d1(orc):
    q = np.array([0.3, -1.1, 0.7]).reshape(1, 1, 3, 1)
    k = np.array([0.1, 0.5, -0.4]).reshape(1, 1, 3, 1)
    v = np.array([1.0, 2.0, -3.0]).reshape(1, 1, 3, 1)
    w = 0.9
    out, den = orc.fwd(q, k, v, np.array([[[w]]]), None, causal=True)
    A = np.cos(w * (q.reshape(3, 1) - k.reshape(1, 3))) * np.tril(np.ones((3, 3)))
    assert np.allclose(den[0, 0], A.sum(1), rtol=1e-14, atol=0), "closed form den"
    assert np.allclose(out[0, 0, :, 0], A @ v.reshape(3) / A.sum(1), rtol=1e-13), "closed form"


def pin_causal_last_equals_noncausal(orc):
    for variant in ("s", "n"):
        q, k, v, W1, W2 = _case(20, 2, 2, 33, 4, 6, variant)
        oc, dc = orc.fwd(q, k, v, W1, W2, True)
        on, dn = orc.fwd(q, k, v, W1, W2, False)
        assert _rel(oc[:, :, -1], on[:, :, -1]) < 1e-12, "causal last != non-causal"
        assert _rel(dc[:, :, -1], dn[:, :, -1]) < 1e-12, "causal last den != non-causal"


def pin_first_and_constant(orc):
    for variant in ("s", "n"):
        q, k, v, W1, W2 = _case(21, 2, 2, 19, 4, 6, variant)
        out, _ = orc.fwd(q, k, v, W1, W2, True)
        assert _rel(out[:, :, 0], v[:, :, 0]) < 1e-13, "causal O_0 != v_0"
        for causal in (True, False):
            c = np.full_like(v, 1.75)
            out, _ = orc.fwd(q, k, c, W1, W2, causal)
            assert np.allclose(out, 1.75, rtol=1e-12, atol=0), "constant v not preserved"


def _loss(q, k, v, W1, W2, causal, dO):
    return float(np.sum(brute.attention(q, k, v, W1, W2, causal)[0] * dO))


def pin_finite_differences(orc):
    h = 1e-6
    for variant in ("s", "n"):
        for causal in (True, False):
            q, k, v, W1, W2 = _case(30, 2, 2, 5, 3, 4, variant)
            dO = _rng(31).standard_normal(q.shape)
            grads = orc.bwd(q, k, v, W1, W2, causal, dO)
            params = [q, k, v, W1] + ([W2] if W2 is not None else [])
            for idx, (p, gp) in enumerate(zip(params, grads)):
                fd = np.zeros_like(p)
                it = np.nditer(p, flags=["multi_index"])
                for _ in it:
                    mi = it.multi_index
                    old = p[mi]
                    p[mi] = old + h
                    lp = _loss(q, k, v, W1, W2, causal, dO)
                    p[mi] = old - h
                    lm = _loss(q, k, v, W1, W2, causal, dO)
                    p[mi] = old
                    fd[mi] = (lp - lm) / (2 * h)
                err = np.linalg.norm(gp - fd) / np.linalg.norm(fd)
                assert err < 1e-6, f"FD {variant} causal={causal} grad #{idx}: {err:.2e}"


def pin_gradient_invariants(orc):
    for variant in ("s", "n"):
        for causal in (True, False):
            q, k, v, W1, W2 = _case(40, 2, 3, 23, 5, 7, variant)
            dO = _rng(41).standard_normal(q.shape)
            dq, dk, dv, dW1, dW2 = orc.bwd(q, k, v, W1, W2, causal, dO)
            s_dv, s_do = dv.sum(axis=2), dO.sum(axis=2)
            assert _rel(s_dv, s_do) < 1e-11, "sum dv != sum dO"
            lhs = np.sum(dW1 * W1) + (np.sum(dW2 * W2) if W2 is not None else 0.0)
            rhs = np.sum(dq * q) + np.sum(dk * k)
            assert abs(lhs - rhs) < 1e-10 * max(abs(rhs), 1.0), "Euler identity"
            if variant == "s":
                t = dq.sum(axis=2) + dk.sum(axis=2)
                scale = np.abs(dq).sum(axis=2) + np.abs(dk).sum(axis=2)
                assert np.all(np.abs(t) < 1e-11 * scale), "translation invariance"


# -------------------------------------------------------------------------------------
# The norm prefactor of Sec. 3.2: phi~(x) = exp(|x|^2 / exp(tau)) phi(x), tau per head.
# The numpy N x N form applies it literally to queries and keys; the C linear form keeps
# only the key weight (the query factor cancels row by row).
# -------------------------------------------------------------------------------------
_TAU = np.array([1.0, 2.5])


def _qfactor(q, tau):
    return np.exp(np.sum(q * q, axis=-1) / np.exp(tau)[:, None])


def pin_prefactor_linear_equals_brute(orc):
    for variant in ("s", "n"):
        for causal in (True, False):
            for N in (1, 3, 17, 64):
                q, k, v, W1, W2 = _case(50 + N, 2, 2, N, 5, 7, variant)
                out, den = orc.fwd(q, k, v, W1, W2, causal, tau=_TAU)
                bo, bd = brute.attention(q, k, v, W1, W2, causal, tau=_TAU)
                assert _rel(out, bo) < 1e-11, f"prefactor out {variant} causal={causal} N={N}"
                assert _rel(den * _qfactor(q, _TAU), bd) < 1e-12, f"prefactor den {variant}"


def pin_prefactor_vanishes_as_tau_grows(orc):
    """exp(-tau) -> 0: the weights tend to 1 (tau = 80 makes them 1 in fp64)."""
    for variant in ("s", "n"):
        q, k, v, W1, W2 = _case(60, 2, 2, 11, 5, 7, variant)
        o0, d0 = orc.fwd(q, k, v, W1, W2, True)
        o1, d1 = orc.fwd(q, k, v, W1, W2, True, tau=np.array([80.0, 80.0]))
        assert np.array_equal(o0, o1) and np.array_equal(d0, d1), "tau -> inf limit"


def pin_prefactor_equal_key_norms(orc):
    """Keys of one norm r: every weight is exp(r^2 exp(-tau)), a common factor, so O is
    the output without the prefactor and den is that factor times its den."""
    for variant in ("s", "n"):
        for causal in (True, False):
            q, k, v, W1, W2 = _case(61, 2, 2, 13, 5, 7, variant)
            k = k / np.linalg.norm(k, axis=-1, keepdims=True) * 1.3
            o0, d0 = orc.fwd(q, k, v, W1, W2, causal)
            o1, d1 = orc.fwd(q, k, v, W1, W2, causal, tau=_TAU)
            w = np.exp(1.3 ** 2 / np.exp(_TAU))[None, :, None]
            assert _rel(o1, o0) < 1e-13, "equal key norms: O changed"
            assert _rel(d1, w * d0) < 1e-13, "equal key norms: den not scaled"


def _loss_tau(q, k, v, W1, W2, causal, dO, tau):
    return float(np.sum(brute.attention(q, k, v, W1, W2, causal, tau=tau)[0] * dO))


def pin_prefactor_finite_differences(orc):
    h = 1e-6
    for variant in ("s", "n"):
        for causal in (True, False):
            q, k, v, W1, W2 = _case(62, 2, 2, 5, 3, 4, variant)
            tau = _TAU.copy()
            dO = _rng(63).standard_normal(q.shape)
            grads = orc.bwd(q, k, v, W1, W2, causal, dO, tau=tau)
            params = [q, k, v, W1] + ([W2] if W2 is not None else [])
            pg = list(zip(params, grads[:len(params)])) + [(tau, grads[5])]
            for idx, (p, gp) in enumerate(pg):
                fd = np.zeros_like(p)
                it = np.nditer(p, flags=["multi_index"])
                for _ in it:
                    mi = it.multi_index
                    old = p[mi]
                    p[mi] = old + h
                    lp = _loss_tau(q, k, v, W1, W2, causal, dO, tau)
                    p[mi] = old - h
                    lm = _loss_tau(q, k, v, W1, W2, causal, dO, tau)
                    p[mi] = old
                    fd[mi] = (lp - lm) / (2 * h)
                err = np.linalg.norm(gp - fd) / np.linalg.norm(fd)
                assert err < 1e-6, f"prefactor FD {variant} causal={causal} #{idx}: {err:.2e}"


def pin_prefactor_scaling_identity(orc):
    """x -> l x, W -> W / l, tau -> tau + 2 ln l leaves every output unchanged, so per head
    <dW1, W1> + <dW2, W2> = sum <dq, q> + <dk, k> + 2 dtau; rows of weights still sum to 1."""
    for variant in ("s", "n"):
        for causal in (True, False):
            q, k, v, W1, W2 = _case(64, 2, 2, 19, 5, 7, variant)
            dO = _rng(65).standard_normal(q.shape)
            dq, dk, dv, dW1, dW2, dtau = orc.bwd(q, k, v, W1, W2, causal, dO, tau=_TAU)
            assert _rel(dv.sum(axis=2), dO.sum(axis=2)) < 1e-11, "prefactor: sum dv != sum dO"
            lhs = np.sum(dW1 * W1, axis=(1, 2))
            if W2 is not None:
                lhs = lhs + np.sum(dW2 * W2, axis=(1, 2))
            rhs = np.sum(dq * q, axis=(0, 2, 3)) + np.sum(dk * k, axis=(0, 2, 3)) + 2 * dtau
            assert np.all(np.abs(lhs - rhs) < 1e-10 * np.maximum(np.abs(rhs), 1.0)), \
                "prefactor scaling identity"


def pin_prefactor_decode(orc):
    for variant in ("s", "n"):
        B, H, N, d, M = 2, 2, 9, 5, 7
        q, k, v, W1, W2 = _case(66, B, H, N, d, M, variant)
        bo, _ = brute.attention(q, k, v, W1, W2, True, tau=_TAU)
        S = np.zeros((B, H, 2 * M, d))
        z = np.zeros((B, H, 2 * M))
        for i in range(N):
            out, _, S, z = orc.decode(q[:, :, i], k[:, :, i], v[:, :, i], W1, W2, S, z,
                                      tau=_TAU)
            assert _rel(out, bo[:, :, i]) < 1e-11, f"prefactor decode {variant} i={i}"


# -------------------------------------------------------------------------------------
# Attention-weight distillation loss (the appendix's distillation setting).
# -------------------------------------------------------------------------------------
def pin_awd_equals_brute(orc):
    """The C loss equals the numpy form with explicit P and R, the prefactor on queries
    and keys as printed (so the query factor's cancellation is checked too)."""
    for variant in ("s", "n"):
        for causal in (False, True):
            for N in (1, 3, 17, 64):
                for tau in (None, _TAU):
                    q, k, _, W1, W2 = _case(70 + N, 2, 2, N, 5, 7, variant)
                    a = orc.awd(q, k, W1, W2, causal, tau=tau)
                    b = brute.awd_loss(q, k, W1, W2, causal, tau=tau)
                    assert _rel(a, b) < 1e-12, f"awd {variant} causal={causal} N={N}"


def pin_awd_single_key(orc):
    """One key: P = R = 1, so the loss is 0 exactly; causally the first query adds 0."""
    q, k, _, W1, W2 = _case(71, 2, 2, 1, 5, 7, "n")
    assert np.all(orc.awd(q, k, W1, W2) == 0.0), "awd N=1"


def pin_awd_closed_form_d1(orc):
    """d = 1, M = 1, stationary: A_ij is proportional to cos(w (q_i - k_j)) and the teacher
    is softmax_j(q_i k_j)."""
    q = np.array([0.3, -0.4, 0.2, 0.5]).reshape(1, 1, 4, 1)
    k = np.array([0.1, 0.25, -0.3, 0.0]).reshape(1, 1, 4, 1)
    w = 0.7
    L = orc.awd(q, k, np.array([[[w]]]), None, causal=False)[0, 0]
    qq, kk = q.reshape(4, 1), k.reshape(1, 4)
    P = np.exp(qq * kk) / np.exp(qq * kk).sum(axis=1, keepdims=True)
    A = np.cos(w * (qq - kk))
    R = A / A.sum(axis=1, keepdims=True)
    assert abs(L - (-np.sum(P * np.log(R)) / 4)) < 1e-14, "awd closed form"


def pin_awd_gibbs(orc):
    """Cross-entropy >= entropy: L >= mean_i H(P_i) (all kernel entries positive here)."""
    for variant in ("s", "n"):
        for causal in (False, True):
            q, k, _, W1, W2 = _case(72, 2, 3, 29, 6, 9, variant)
            L = orc.awd(q, k, W1, W2, causal)
            s = np.einsum("bhid,bhjd->bhij", q, k) / np.sqrt(6)
            if causal:
                s = np.where(np.tril(np.ones((29, 29), bool)), s, -np.inf)
            P = np.exp(s - s.max(-1, keepdims=True))
            P /= P.sum(-1, keepdims=True)
            Hp = -np.sum(np.where(P > 0, P * np.log(np.where(P > 0, P, 1.0)), 0.0), axis=(-1, -2)) / 29
            assert np.all(L >= Hp - 1e-12), "awd below the teacher's entropy"


def pin_awd_equal_key_norms(orc):
    """Keys of one norm make the prefactor a common factor of R: the loss is unchanged."""
    q, k, _, W1, W2 = _case(73, 2, 2, 21, 5, 7, "n")
    k = k / np.linalg.norm(k, axis=-1, keepdims=True) * 1.1
    assert _rel(orc.awd(q, k, W1, W2, tau=_TAU), orc.awd(q, k, W1, W2)) < 1e-13, "awd tau"


def pin_awd_nonpositive_entries(orc):
    """Large frequencies and few of them make some kernel estimates and some row sums
    negative; entries with a non-positive normalised weight count log 1e-6, as in the
    numpy form."""
    q, k, _, W1, W2 = _case(74, 1, 2, 23, 5, 3, "s", qk_scale=2.0)
    W1 = W1 * 4.0
    K = brute.kernel_matrix(q, k, W1)
    assert np.any(K <= 0) and np.any(K.sum(-1) < 0), "the case needs both kinds"
    assert _rel(orc.awd(q, k, W1), brute.awd_loss(q, k, W1)) < 1e-12, "awd clamp"


# -------------------------------------------------------------------------------------
# Gradient of the distillation loss with respect to the kernel's parameters (W1, W2,
# tau): the distillation trains only the feature map, q and k are frozen.
# -------------------------------------------------------------------------------------
def _awd_case(variant):
    """Small case with negative kernel estimates (and, for s, negative row sums) but no
    normalised weight near 0, so central differences do not straddle the clamp."""
    seed = 124 if variant == "s" else 109
    q, k, _, W1, W2 = _case(seed, 2, 2, 6, 3, 4, variant, qk_scale=1.0)
    return q, k, W1 * 1.5, None if W2 is None else W2 * 1.5


def pin_awd_grad_finite_differences(orc):
    """dW1, dW2, dtau against central differences of the numpy explicit-matrix loss
    (sum form of the nonstationary features, prefactor on queries and keys as printed),
    weighted by a random upstream gradient per sequence."""
    h = 1e-6
    dl = _rng(75).standard_normal((2, 2))
    for variant in ("s", "n"):
        q, k, W1, W2 = _awd_case(variant)
        K = brute.kernel_matrix(q, k, W1, W2)
        assert np.any(K < 0), "the case needs negative kernel entries"
        for causal in (False, True):
            for tau in (None, _TAU.copy()):
                def total():
                    return float(np.sum(dl * brute.awd_loss(q, k, W1, W2, causal, tau=tau)))
                grads = orc.awd_bwd(q, k, W1, W2, causal, tau=tau, dloss=dl)
                params = [(W1, grads[0])]
                if W2 is not None:
                    params.append((W2, grads[1]))
                if tau is not None:
                    params.append((tau, grads[2]))
                for idx, (p, gp) in enumerate(params):
                    fd = np.zeros_like(p)
                    it = np.nditer(p, flags=["multi_index"])
                    for _ in it:
                        mi = it.multi_index
                        old = p[mi]
                        p[mi] = old + h
                        lp = total()
                        p[mi] = old - h
                        lm = total()
                        p[mi] = old
                        fd[mi] = (lp - lm) / (2 * h)
                    err = np.linalg.norm(gp - fd) / np.linalg.norm(fd)
                    assert err < 1e-6, (f"awd grad FD {variant} causal={causal} "
                                        f"tau={tau is not None} #{idx}: {err:.2e}")


def pin_awd_grad_closed_form_d1(orc):
    """d = 1, M = 1, stationary: A_ij is proportional to cos(w D_ij), D_ij = q_i - k_j, so
    dL/dw = -(1/N) sum_i [ sum_j P_ij (-D_ij tan(w D_ij))  -  c_i (sum_j -D_ij sin(w D_ij))
    / (sum_j cos(w D_ij)) ]  with every entry positive here (c_i = 1), written out."""
    q = np.array([0.3, -0.4, 0.2, 0.5]).reshape(1, 1, 4, 1)
    k = np.array([0.1, 0.25, -0.3, 0.0]).reshape(1, 1, 4, 1)
    w = 0.7
    for causal in (False, True):
        dW1, _, _ = orc.awd_bwd(q, k, np.array([[[w]]]), None, causal)
        qq, kk = q.reshape(4, 1), k.reshape(1, 4)
        Dl = qq - kk
        mask = np.tril(np.ones((4, 4), bool)) if causal else np.ones((4, 4), bool)
        s = np.where(mask, qq * kk, -np.inf)
        P = np.exp(s - s.max(1, keepdims=True))
        P /= P.sum(1, keepdims=True)
        A = np.where(mask, np.cos(w * Dl), 0.0)
        dA = np.where(mask, -Dl * np.sin(w * Dl), 0.0)
        assert np.all(A[mask] > 0), "the case needs positive weights"
        g = np.sum(P * np.where(mask, dA / np.where(mask, A, 1.0), 0.0), 1) - (
            dA.sum(1) / A.sum(1))
        assert abs(dW1[0, 0, 0] - (-np.sum(g) / 4)) < 1e-14, "awd grad closed form"


def pin_awd_grad_single_key(orc):
    """One key: R = 1 whatever the parameters, so every gradient is exactly 0."""
    q, k, _, W1, W2 = _case(76, 2, 2, 1, 5, 7, "n")
    dW1, dW2, dtau = orc.awd_bwd(q, k, W1, W2, tau=_TAU)
    assert np.all(dW1 == 0.0) and np.all(dW2 == 0.0) and np.all(dtau == 0.0), "awd grad N=1"


def pin_awd_grad_equal_key_norms(orc):
    """Keys of one norm: the prefactor is a common factor of each row of R, so the loss
    does not depend on tau and dtau = 0 (the -c_i/D_i term must cancel the P/A term)."""
    for causal in (False, True):
        q, k, _, W1, W2 = _case(77, 2, 2, 19, 5, 7, "n")
        k = k / np.linalg.norm(k, axis=-1, keepdims=True) * 1.3
        dW1, _, dtau = orc.awd_bwd(q, k, W1, W2, causal, tau=_TAU)
        assert np.all(np.abs(dtau) < 1e-11 * np.abs(dW1).sum()), "awd dtau, equal norms"
        assert np.abs(dW1).sum() > 1e-6, "the case needs a nonzero gradient"


def pin_awd_grad_tied_frequencies(orc):
    """W2 = W1 reduces Flexformer_n to Flexformer_s at W1, so moving both together is
    moving the stationary frequencies: dW1_n + dW2_n = dW_s."""
    for causal in (False, True):
        q, k, _, W1, _ = _case(78, 2, 2, 13, 5, 7, "s")
        dn1, dn2, _ = orc.awd_bwd(q, k, W1, W1.copy(), causal)
        ds, _, _ = orc.awd_bwd(q, k, W1, None, causal)
        assert _rel(dn1 + dn2, ds) < 1e-12, "awd grad W2 = W1"


ALL_PINS = [
    pin_origin_features, pin_stationary_unit_norm, pin_sum_to_product, pin_w2_equals_w1,
    pin_bochner, pin_yaglom, pin_linear_equals_brute, pin_decode_equals_brute,
    pin_closed_form_d1,
    pin_causal_last_equals_noncausal, pin_first_and_constant, pin_finite_differences,
    pin_gradient_invariants, pin_prefactor_linear_equals_brute,
    pin_prefactor_vanishes_as_tau_grows, pin_prefactor_equal_key_norms,
    pin_prefactor_finite_differences, pin_prefactor_scaling_identity, pin_prefactor_decode,
    pin_awd_equals_brute, pin_awd_single_key, pin_awd_closed_form_d1, pin_awd_gibbs,
    pin_awd_equal_key_norms, pin_awd_nonpositive_entries, pin_awd_grad_finite_differences,
    pin_awd_grad_single_key, pin_awd_grad_equal_key_norms, pin_awd_grad_tied_frequencies,
    pin_awd_grad_closed_form_d1,
]
