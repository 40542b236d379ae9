"""The block factorisation of Eq. (1) that the chunked form computes, checked in FP64 against
the oracle's token-by-token recurrence.

Within a block of L tokens starting from state S_b (rows = key channels), with
d_t = e^{-s_t}, Dc_t = d_0 ... d_t (per key row) and u_t = w_t * v_t - (D_t S_{t-1})^T a_t:

    p_t = S_b^T (a_t * Dc_t) + sum_{s<t}  A_ts u_s,   A_ts = sum_i a_ti k_si Dc_ti / Dc_si
    o_t = S_b^T (q_t * Dc_t) + sum_{s<=t} M_ts u_s,   M_ts = sum_i q_ti k_si Dc_ti / Dc_si
    S_e = Dc_{L-1} * S_b + sum_t (k_t * Dc_{L-1} / Dc_t) u_t^T

Unrolling Eq. (1) over the block gives these identities exactly; the tests restate them in
numpy (independent of the oracle's C code and of the CUDA kernels) so that a wrong index, a
dropped diagonal or a mis-placed decay factor in the reading fails here, on the CPU.
"""
import numpy as np
import pytest


def _block_form(S0, k, q, v, s, a, w, L, a_diag=-1, m_diag=0):
    """FP64 readouts and end state of Eq. (1) computed block by block (blocks of L tokens,
    the last one ragged).  ``a_diag`` / ``m_diag``: the highest diagonal kept in A and M
    (-1: s < t, 0: s <= t); other values exist only to show that the check has teeth."""
    k, q, v, s, a, w = (x.astype(np.float64) for x in (k, q, v, s, a, w))
    T = k.shape[0]
    S = np.array(S0, dtype=np.float64)
    o = np.zeros((T, v.shape[1]))
    for t0 in range(0, T, L):
        t1 = min(t0 + L, T)
        Dc = np.exp(-np.cumsum(s[t0:t1], axis=0))          # (n, dk): Dc_t = d_0 ... d_t
        kb, qb, ab = k[t0:t1], q[t0:t1], a[t0:t1]
        Kt, Qt, Kh = ab * Dc, qb * Dc, kb / Dc
        A = np.tril(Kt @ Kh.T, a_diag)                       # strictly lower: s < t
        M = np.tril(Qt @ Kh.T, m_diag)                       # with the diagonal: s <= t
        n = t1 - t0
        u = np.zeros((n, v.shape[1]))
        base = Kt @ S                                        # rows: (S_b^T (a_t Dc_t))^T
        for t in range(n):                                   # forward substitution
            u[t] = (w[t0 + t] * v[t0 + t] - (base[t] + A[t, :t] @ u[:t])) / (1.0 + A[t, t])
        o[t0:t1] = Qt @ S + M @ u
        Kbar = kb * Dc[-1] / Dc                              # k_t Dc_{L-1} / Dc_t
        S = Dc[-1][:, None] * S + Kbar.T @ u
    return o, S


def _inputs(rng, T, dk, dv, erase, rate_hi=0.4):
    k = rng.standard_normal((T, dk)).astype(np.float32)
    k /= np.linalg.norm(k, axis=1, keepdims=True)
    q = (rng.standard_normal((T, dk)) / np.sqrt(dk)).astype(np.float32)
    v = rng.standard_normal((T, dv)).astype(np.float32)
    s = rng.uniform(0.0, rate_hi, (T, dk)).astype(np.float32)
    if erase:
        beta = rng.uniform(0.1, 1.0, T).astype(np.float32)
        a = (beta[:, None] * k).astype(np.float32)
        w = np.repeat(beta[:, None], dv, axis=1).astype(np.float32)
    else:
        a = np.zeros_like(k)
        w = np.ones((T, dv), np.float32)
    return k, q, v, s, a, w


@pytest.mark.parametrize("T,L", [(64, 16), (40, 16), (16, 16), (5, 16), (37, 8), (1, 16)])
@pytest.mark.parametrize("erase", [True, False])
def test_block_form_equals_token_recurrence(orc, T, L, erase):
    """Whole, ragged and single-token blocks, with the delta rule (a = beta k, w = beta) and
    without erasure (a = 0, w = 1): readouts and end state equal the FP64 token loop."""
    rng = np.random.default_rng(1000 + 7 * T + L + erase)
    dk, dv = 24, 20
    S0 = rng.standard_normal((dk, dv))
    args = _inputs(rng, T, dk, dv, erase)
    o_ref, S_ref = orc.recur(S0, *args, dtype=np.float64)
    o, S = _block_form(S0, *args, L)
    assert np.allclose(o, o_ref, rtol=1e-11, atol=1e-12)
    assert np.allclose(S, S_ref, rtol=1e-11, atol=1e-12)


def test_block_form_general_erasure(orc):
    """The identities hold for any a and w of Eq. (1), not only a = beta k."""
    rng = np.random.default_rng(77)
    T, dk, dv = 48, 16, 12
    k, q, v, s, _, _ = _inputs(rng, T, dk, dv, True)
    a = (0.3 * rng.standard_normal((T, dk))).astype(np.float32)
    w = rng.uniform(0.2, 1.5, (T, dv)).astype(np.float32)
    S0 = rng.standard_normal((dk, dv))
    o_ref, S_ref = orc.recur(S0, k, q, v, s, a, w, dtype=np.float64)
    o, S = _block_form(S0, k, q, v, s, a, w, 16)
    assert np.allclose(o, o_ref, rtol=1e-11, atol=1e-12)
    assert np.allclose(S, S_ref, rtol=1e-11, atol=1e-12)


def test_block_form_detects_a_misplaced_diagonal(orc):
    """The check has teeth: taking the diagonal into A (p_t reading u_t) or out of M (o_t
    missing its own write) moves the readouts far beyond rounding."""
    rng = np.random.default_rng(5)
    T, dk, dv = 32, 16, 8
    args = _inputs(rng, T, dk, dv, True)
    S0 = rng.standard_normal((dk, dv))
    o_ref, _ = orc.recur(S0, *args, dtype=np.float64)
    for a_diag, m_diag in ((0, 0), (-1, -1)):
        o_bad, _ = _block_form(S0, *args, 16, a_diag, m_diag)
        assert not np.allclose(o_bad, o_ref, rtol=1e-3, atol=1e-3)


def test_block_decay_factor_range(orc):
    """Why the chunked form needs every row's decay over one block to stay a normal FP32
    number: k / Dc overflows FP32 once the rates over 16 tokens sum past about 87, while
    the FP64 factorisation and the token loop still agree."""
    rng = np.random.default_rng(9)
    T, dk, dv = 16, 8, 4
    k, q, v, s, a, w = _inputs(rng, T, dk, dv, True)
    s[:, 0] = 6.0                                            # 96 over the block on row 0
    Dc32 = np.exp(-np.cumsum(s.astype(np.float32), axis=0, dtype=np.float32))
    assert Dc32[-1, 0] < np.finfo(np.float32).tiny           # below the normal range
    with np.errstate(over="ignore", divide="ignore"):
        assert not np.all(np.isfinite(k.astype(np.float32) / Dc32))
    S0 = rng.standard_normal((dk, dv))
    o_ref, S_ref = orc.recur(S0, k, q, v, s, a, w, dtype=np.float64)
    o, S = _block_form(S0, k, q, v, s, a, w, 16)
    assert np.allclose(o, o_ref, rtol=1e-9, atol=1e-12)
    assert np.allclose(S, S_ref, rtol=1e-9, atol=1e-12)
