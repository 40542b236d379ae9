"""FP64 theory of the method, written from the paper (test infrastructure only).

Sec. 2 (Proposition 1, Eq. 2), the erasure approximation, and Sec. 3 (Eq. 3, Eq. 4, the
AM/GM gain, the persistence factors of the ablations).  Plain numpy in float64.
"""
from __future__ import annotations

import numpy as np


def propagation_matrix(k, a, s):
    """F_t = (I - k a^T) diag(e^{-s}) (Sec. 2, between write-backs)."""
    k = np.asarray(k, np.float64)
    a = np.asarray(a, np.float64)
    s = np.broadcast_to(np.asarray(s, np.float64), k.shape)
    return (np.eye(k.size) - np.outer(k, a)) @ np.diag(np.exp(-s))


def gramian_exact(F, q, C, taus, tol=1e-14, max_lag=None):
    """Eq. (2) on a realised sequence.

    ``F[t]`` is F_t (dk x dk) and ``q[t]`` the query at token t, for t = 0..T-1.  For each
    write-back position tau in ``taus`` the error injected there is read at tau + l for
    l >= 1 through Phi_l = F_{tau+l} ... F_{tau+1}:  sum_l (Phi_l^T q_{tau+l})_i^2.  The
    sum stops when the propagated energy falls below ``tol`` of what has accumulated, or at
    the end of the sequence.  Averaging over tau and dividing by C gives Gamma_i.
    """
    F = np.asarray(F, np.float64)
    q = np.asarray(q, np.float64)
    T, dk = q.shape
    acc = np.zeros(dk)
    for tau in taus:
        Phi = np.eye(dk)
        tot = np.zeros(dk)
        for ell in range(1, T - tau):
            if max_lag is not None and ell > max_lag:
                break
            Phi = F[tau + ell] @ Phi
            contrib = (Phi.T @ q[tau + ell]) ** 2
            tot += contrib
            if np.all(Phi == 0) or (ell > 8 and np.max(np.sum(Phi ** 2, axis=0)) < tol):
                break
        acc += tot
    return acc / (len(taus) * C)


def gramian_expected_const(F, Q, C, tol=1e-15, max_lag=100000):
    """Eq. (2) for a constant F and E[q q^T] = Q: Gamma_i = (1/C) sum_l (F^l^T Q F^l)_ii."""
    F = np.asarray(F, np.float64)
    dk = F.shape[0]
    Phi = np.eye(dk)
    tot = np.zeros(dk)
    for _ in range(max_lag):
        Phi = F @ Phi
        c = np.einsum("mi,mn,ni->i", Phi, Q, Phi)
        tot += c
        if np.max(np.abs(c)) < tol * max(1.0, np.max(tot)):
            break
    return tot / C


def gamma_closed_form(rho, s, C):
    """Prop. 1, constant diagonal decay without erasure: rho_i / (C expm1(2 s_i))."""
    return np.asarray(rho, np.float64) / (C * np.expm1(2.0 * np.asarray(s, np.float64)))


def gamma_bound(Eq2, s, C):
    """Prop. 1, constant per-head decay with a = beta k, beta in [0, 2]:
    Gamma_i <= E|q|^2 / (C expm1(2 s))."""
    return Eq2 / (C * np.expm1(2.0 * s))


def erasure_rate(beta, k_i):
    """Sec. 2, "Approximate erasure rate": r_i = 1/2 E[beta (2 - beta) k_i^2] (per sample)."""
    beta = np.asarray(beta, np.float64)
    return 0.5 * np.mean(beta * (2.0 - beta) * np.asarray(k_i, np.float64) ** 2)


def gamma_approx(rho, s, r, C):
    """Gamma_i ~ rho_i / (C expm1(2 (s_i + r_i)))."""
    return np.asarray(rho, np.float64) / (C * np.expm1(2.0 * (np.asarray(s) + np.asarray(r))))


def gamma_hat(s_hat, r):
    """Eq. (3): Gamma_hat_i = 1 / expm1(2 (s_hat_i + r_i))."""
    return 1.0 / np.expm1(2.0 * (np.asarray(s_hat, np.float64) + np.asarray(r, np.float64)))


def s_hat_from_ema(ema_decay_sq):
    """Sec. 3: s_hat = -1/2 log EMA(e^{2 g}) with g = -s, i.e. of the squared decay factor."""
    return -0.5 * np.log(np.asarray(ema_decay_sq, np.float64))


def alloc_real(c, bbar):
    """Eq. (4): b_i = bbar + 1/2 log2(c_i / GM(c))."""
    c = np.asarray(c, np.float64)
    return bbar + 0.5 * (np.log2(c) - np.mean(np.log2(c)))


def proxy(c, b):
    """The high-rate proxy sum_i c_i 2^{-2 b_i}."""
    return float(np.sum(np.asarray(c, np.float64) * 2.0 ** (-2.0 * np.asarray(b, np.float64))))


def am_gm_gain(c):
    """Sec. 3: distortion reduction over uniform allocation = AM(c) / GM(c)."""
    c = np.asarray(c, np.float64)
    return float(np.mean(c) / np.exp(np.mean(np.log(c))))


def w1(a):
    """DAMP's uncapped persistence 1 / (1 - a^2) for effective decay a (Sec. 1)."""
    return 1.0 / (1.0 - np.asarray(a, np.float64) ** 2)


def h_C(s, C):
    """Table 1's write-back factor h^(C) = 1 / (1 - e^{-2 C s})."""
    return 1.0 / (1.0 - np.exp(-2.0 * C * np.asarray(s, np.float64)))
