"""Pins of the FP64 theory (Sec. 2 Prop. 1 / Eq. 2, erasure approximation; Sec. 3 Eq. 3-4)
against what the paper and the mathematics fix: closed forms, the printed worked example,
a norm bound, the DAMP identity and a Monte Carlo noise-injection experiment run through the
oracle's independent recurrence code."""
import math
import os

import numpy as np
import pytest

from oracle import theory as th

GOLD = os.path.join(os.path.dirname(__file__), "golden")


def _read_kv(name):
    out = {}
    for line in open(os.path.join(GOLD, name)):
        line = line.strip()
        if line and not line.startswith("#"):
            k, v = line.split()
            out[k] = float(v)
    return out


def _sig(x, n):
    return float(f"{x:.{n}g}")


def test_erasure_worked_example_matches_printed_values():
    """Sec. 2 'Approximate erasure rate': exact 24.9, approximate 2.06."""
    g = _read_kv("erasure_example.txt")
    dk = int(g["dk"])
    k = np.ones(dk) / math.sqrt(dk)
    a = g["beta"] * k
    F = th.propagation_matrix(k, a, np.full(dk, g["s"]))
    exact = th.gramian_expected_const(F, np.eye(dk), int(g["C"]))
    r = th.erasure_rate([g["beta"]], k[0])
    approx = th.gamma_approx(1.0, g["s"], r, int(g["C"]))
    n = int(g["sig_figs"])
    assert _sig(exact[0], n) == g["gamma_exact"]
    assert _sig(exact[1], n) == g["gamma_exact"]
    assert _sig(approx, n) == g["gamma_approx"]
    # brute force: explicit matrix powers, independent of the helper above
    tot = sum(np.trace(np.linalg.matrix_power(F, l).T @ np.linalg.matrix_power(F, l)) / dk
              for l in range(1, 4000))
    assert abs(tot - exact[0]) < 1e-9


@pytest.mark.parametrize("C", [1, 4, 16])
def test_gramian_constant_decay_closed_form(C):
    """Prop. 1: constant diagonal decay, no erasure -> Gamma_i = rho_i / (C expm1(2 s_i))."""
    rng = np.random.default_rng(1)
    dk = 5
    s = rng.uniform(0.02, 0.5, dk)
    F = np.diag(np.exp(-s))
    T = 4000
    # constant query: exact up to the truncation e^{-2 s T}
    qc = rng.standard_normal(dk)
    G = th.gramian_exact([F] * T, np.tile(qc, (T, 1)), C, taus=[0])
    assert np.allclose(G, th.gamma_closed_form(qc ** 2, s, C), rtol=1e-12, atol=0)
    # expectation form with E[q q^T] = diag(rho)
    rho = rng.uniform(0.5, 2.0, dk)
    G2 = th.gramian_expected_const(F, np.diag(rho), C)
    assert np.allclose(G2, th.gamma_closed_form(rho, s, C), rtol=1e-10)


def test_gramian_random_queries_monte_carlo_ci():
    """Random queries: realised Eq. (2) averaged over many write-backs lies within the
    Monte Carlo interval of the closed form."""
    rng = np.random.default_rng(2)
    dk, C, T = 4, 2, 6000
    s = np.array([0.05, 0.1, 0.3, 1.0])
    rho = np.array([1.0, 0.5, 2.0, 1.5])
    q = rng.standard_normal((T, dk)) * np.sqrt(rho)
    F = [np.diag(np.exp(-s))] * T
    taus = list(range(C - 1, T - 400, C))
    G = th.gramian_exact(F, q, C, taus)
    ref = th.gamma_closed_form(rho, s, C)
    # per-write-back samples are correlated over ~1/s lags; a loose 10% band at T = 6000
    assert np.all(np.abs(G / ref - 1) < 0.1)


def test_gramian_bound_with_erasure():
    """Prop. 1: constant per-head decay, a = beta k, beta in [0, 2], unit keys and queries:
    Gamma_i <= E|q|^2 / (C expm1(2 s)) -- holds for every realisation."""
    rng = np.random.default_rng(3)
    dk, T, s = 6, 3000, 0.02
    for C in (1, 8):
        k = rng.standard_normal((T, dk))
        k /= np.linalg.norm(k, axis=1, keepdims=True)
        beta = rng.uniform(0, 2, T)
        q = rng.standard_normal((T, dk))
        q /= np.linalg.norm(q, axis=1, keepdims=True)
        F = [th.propagation_matrix(k[t], beta[t] * k[t], s) for t in range(T)]
        G = th.gramian_exact(F, q, C, taus=list(range(C - 1, T // 2, C)))
        assert np.all(G <= th.gamma_bound(1.0, s, C) * (1 + 1e-12))
        assert np.all(G > 0)


def test_damp_identity_no_erasure():
    """Sec. 1/3: without erasure Gamma_hat = w1(e^{-s}) e^{-2s} = 1/expm1(2s)."""
    s = np.logspace(-4, 1, 200)
    lhs = th.gamma_hat(s, 0.0)
    rhs = th.w1(np.exp(-s)) * np.exp(-2 * s)
    assert np.allclose(lhs, rhs, rtol=1e-10)
    # and the write-back factor of Table 1 tends to w1 at C = 1
    assert np.allclose(th.h_C(s, 1), th.w1(np.exp(-s)), rtol=1e-12)


@pytest.mark.parametrize("C", [1, 4])
def test_prop1_noise_injection_monte_carlo(orc, C):
    """Prop. 1 / Eq. (2): zero-mean noise of row variance sigma_i^2 injected at every
    write-back of a tiny KDA-style recurrence gives a time-averaged readout MSE per value
    column of sum_i Gamma_i sigma_i^2.  The readouts come from the oracle's own recurrence
    code (independent of the Gramian helper); by linearity the noise alone is propagated
    (zero writes, zero initial state)."""
    rng = np.random.default_rng(10 + C)
    dk = dv = 4
    T = 160
    nwb = T // C
    k = rng.standard_normal((T, dk))
    k /= np.linalg.norm(k, axis=1, keepdims=True)
    beta = rng.uniform(0.2, 1.5, T)
    s = rng.uniform(0.01, 0.4, (T, dk))           # per-row decay: F is not symmetric
    q = rng.standard_normal((T, dk))
    a = beta[:, None] * k
    sigma = np.array([1.0, 0.5, 2.0, 0.25])
    F = [th.propagation_matrix(k[t], a[t], s[t]) for t in range(T)]
    taus = [c * C + C - 1 for c in range(nwb)]
    G = th.gramian_exact(F, q, C, taus)
    pred = float(np.sum(G * sigma ** 2))
    f32 = lambda x: np.ascontiguousarray(x, np.float32)
    v0 = np.zeros((C, dv), np.float32)
    w = np.ones((C, dv), np.float32)
    draws = 300
    sq = np.zeros(draws)
    for d in range(draws):
        S = np.zeros((dk, dv))
        acc = 0.0
        for c in range(nwb):
            sl = slice(c * C, c * C + C)
            o, S = orc.recur(S, f32(k[sl]), f32(q[sl]), v0, f32(s[sl]), f32(a[sl]), w,
                             dtype=np.float64)
            acc += float(np.sum(o ** 2))
            S = S + rng.standard_normal((dk, dv)) * sigma[:, None]   # write-back noise
        sq[d] = acc / (T * dv)
    mc, se = sq.mean(), sq.std(ddof=1) / math.sqrt(draws)
    assert abs(mc - pred) < 4 * se + 1e-3 * pred, (mc, pred, se)


@pytest.mark.parametrize("C", [1, 3])
def test_prop1_impulse_responses_equal_gramian(orc, C):
    """Eq. (2) exactly, by linearity: a unit error in row i written back at tau, propagated by
    the oracle's recurrence (zero writes), is read at tau + l as (Phi_l^T q_{tau+l})_i.  The
    summed squared responses must equal C |taus| Gamma_i from the matrix-product helper.  A
    transposed Phi or q, a dropped erase term or an off-by-one lag fails this."""
    rng = np.random.default_rng(20 + C)
    dk, dv, T = 5, 2, 60
    k = rng.standard_normal((T, dk))
    k /= np.linalg.norm(k, axis=1, keepdims=True)
    beta = rng.uniform(0.3, 1.9, T)
    s = rng.uniform(0.01, 0.6, (T, dk))
    q = rng.standard_normal((T, dk))
    a = beta[:, None] * k
    F = [th.propagation_matrix(k[t], a[t], s[t]) for t in range(T)]
    taus = list(range(C - 1, T, C))
    G = th.gramian_exact(F, q, C, taus, tol=0.0)
    f32 = lambda x: np.ascontiguousarray(x, np.float32)
    # the helper works from float64 inputs; feed it the float32-rounded ones the C code sees
    F32 = [th.propagation_matrix(f32(k[t]).astype(np.float64), f32(a[t]).astype(np.float64),
                                 f32(s[t]).astype(np.float64)) for t in range(T)]
    G32 = th.gramian_exact(F32, f32(q).astype(np.float64), C, taus, tol=0.0)
    tot = np.zeros(dk)
    for tau in taus:
        n = T - 1 - tau
        if n == 0:
            continue
        sl = slice(tau + 1, T)
        for i in range(dk):
            S = np.zeros((dk, dv))
            S[i, 0] = 1.0
            o, _ = orc.recur(S, f32(k[sl]), f32(q[sl]), np.zeros((n, dv), np.float32),
                             f32(s[sl]), f32(a[sl]), np.ones((n, dv), np.float32),
                             dtype=np.float64)
            tot[i] += np.sum(o[:, 0] ** 2)
            assert np.all(o[:, 1] == 0)
    assert np.allclose(tot / (len(taus) * C), G32, rtol=1e-9)
    assert np.allclose(G32, G, rtol=1e-5)


def test_real_allocation_budget_and_am_gm_gain():
    """Eq. (4): sum b_i = N bbar exactly; the proxy ratio ours/uniform = GM(c)/AM(c)."""
    rng = np.random.default_rng(4)
    for N, bbar in [(8, 2.0), (128, 4.0), (4096, 3.0)]:
        c = np.exp(rng.normal(0, 2, N))
        b = th.alloc_real(c, bbar)
        assert abs(b.sum() - N * bbar) < 1e-9 * N
        ratio = th.proxy(c, b) / th.proxy(c, np.full(N, bbar))
        assert abs(ratio - 1.0 / th.am_gm_gain(c)) < 1e-10
        # every row ends with the same distortion c_i 4^{-b_i} (the high-rate optimum)
        d = c * 4.0 ** (-b)
        assert np.allclose(d, d[0], rtol=1e-9)
    # uniform weights -> uniform widths and gain 1
    assert np.allclose(th.alloc_real(np.full(7, 3.3), 4.0), 4.0)
    assert abs(th.am_gm_gain(np.full(7, 3.3)) - 1.0) < 1e-12
