"""Pins of the allocation-weight alternatives of Table 1 (weight_kind 1-8) in the oracle.

Each is checked against an identity the paper states or the mathematics fixes: the
write-back factor at C = 1 is the persistence weight; without erasure the weight of Eq. (3) is
the persistence weight times the squared decay (the relation to DAMP in Sec. 1); leaving the
erasure term out equals Eq. (3) when that term is zero; the write-back factor tends to one as
C grows and matches its closed form; shuffling permutes the decay weights without changing
them; range-only and relative-range allocation agree when one group spans the layer.
"""
import numpy as np
import pytest

OURS, RANGE, GAMMA_RAW, NRANGE, PERSIST, WBFACTOR, NOERASE, SHUFFLE, UNIFORM = range(9)


def _stats(N, seed, mr_max=0.3):
    rng = np.random.default_rng(seed)
    ms = rng.uniform(0.01, 0.5, N).astype(np.float32)
    mr = rng.uniform(0.0, mr_max, N).astype(np.float32)
    R = np.exp(rng.normal(0, 0.7, N)).astype(np.float32)
    return ms, mr, R


def _cfg(orc, kind, H=4, dk=32, group_heads=1, C=1, bmin=1, bmax=8, bbar=4):
    return orc.Cfg(B=1, H=H, dk=dk, dv=32, group_heads=group_heads, bbar_num=bbar, bmin=bmin,
                   bmax=bmax, C=C, weight_kind=kind)


def test_write_back_factor_at_c1_is_persistence(orc):
    ms, mr, R = _stats(128, 0)
    w1 = orc.weights(_cfg(orc, PERSIST), ms, mr, R).astype(np.float64)
    h1 = orc.weights(_cfg(orc, WBFACTOR, C=1), ms, mr, R).astype(np.float64)
    assert np.allclose(h1, w1, rtol=2e-6)


def test_no_erasure_weight_is_persistence_times_squared_decay(orc):
    # Gamma_hat with r = 0 is 1/expm1(2 s) = w1 e^{-2s}, and e^{-2 s_hat} = 1 - m_s
    ms, mr, R = _stats(128, 1)
    w1 = orc.weights(_cfg(orc, PERSIST), ms, mr, R).astype(np.float64)
    g0 = orc.weights(_cfg(orc, NOERASE), ms, mr, R).astype(np.float64)
    assert np.allclose(g0, w1 * (1.0 - ms.astype(np.float64)), rtol=4e-7)


def test_no_erasure_equals_eq3_when_erasure_term_is_zero(orc):
    ms, _, R = _stats(128, 2)
    mr0 = np.zeros_like(ms)
    a = orc.weights(_cfg(orc, OURS), ms, mr0, R)
    b = orc.weights(_cfg(orc, NOERASE), ms, np.full_like(ms, 0.2), R)
    assert np.array_equal(a, b)


@pytest.mark.parametrize("C", [2, 3, 16, 64, 1000])
def test_write_back_factor_closed_form(orc, C):
    ms, mr, R = _stats(128, 3)
    rt2 = orc.weights(_cfg(orc, NRANGE), ms, mr, R).astype(np.float64)
    h = orc.weights(_cfg(orc, WBFACTOR, C=C), ms, mr, R).astype(np.float64)
    ref = rt2 / (1.0 - (1.0 - ms.astype(np.float64)) ** C)
    # C FP32 roundings in the power, amplified by 1/(1 - p) when p is near 1
    p = (1.0 - ms.astype(np.float64)) ** C
    tol = 4e-7 * (np.log2(C) + 2) * (1.0 + p / (1.0 - p)) + 4e-7
    assert np.all(np.abs(h - ref) <= tol * ref)


def test_write_back_factor_tends_to_relative_range(orc):
    ms, mr, R = _stats(128, 4)
    rt2 = orc.weights(_cfg(orc, NRANGE), ms, mr, R)
    h = orc.weights(_cfg(orc, WBFACTOR, C=100000), ms, mr, R)
    assert np.array_equal(h, rt2)


@pytest.mark.parametrize("N", [16, 64, 96, 128, 4096, 8192])
def test_shuffle_is_a_bijection(orc, N):
    pi = orc.shuffle_map(N)
    assert np.array_equal(np.sort(pi), np.arange(N))
    if N >= 16:
        assert np.mean(pi == np.arange(N)) < 0.1


def test_shuffle_moves_decay_weights(orc):
    ms, mr, _ = _stats(128, 5)
    R = np.ones(128, np.float32)          # Rtilde = 1: weights are the decay weights alone
    g = orc.weights(_cfg(orc, OURS), ms, mr, R)
    gs = orc.weights(_cfg(orc, SHUFFLE), ms, mr, R)
    assert np.array_equal(np.sort(g), np.sort(gs))
    assert np.array_equal(gs, g[orc.shuffle_map(128)])


def test_raw_range_special_cases(orc):
    ms, mr, R = _stats(128, 6)
    # Gamma_hat = 1 (m_s = 1/2, no erasure): raw range = range alone
    half = np.full(128, 0.5, np.float32)
    zero = np.zeros(128, np.float32)
    assert np.array_equal(orc.weights(_cfg(orc, GAMMA_RAW), half, zero, R),
                          orc.weights(_cfg(orc, RANGE), half, zero, R))
    # unit ranges: raw range = Eq. (3)
    one = np.ones(128, np.float32)
    assert np.array_equal(orc.weights(_cfg(orc, GAMMA_RAW), ms, mr, one),
                          orc.weights(_cfg(orc, OURS), ms, mr, one))


def test_range_and_relative_range_agree_within_one_group(orc):
    # one output-normalisation group spanning the layer: Rtilde^2 = R^2 / const, and a common
    # factor does not change which bits are the most valuable
    ms, mr, R = _stats(128, 7)
    a = orc.alloc(_cfg(orc, RANGE, group_heads=4), ms, mr, R)[0]
    b = orc.alloc(_cfg(orc, NRANGE, group_heads=4), ms, mr, R)[0]
    assert np.array_equal(a, b)
    assert a.sum() == 128 * 4


def test_uniform_weight_gives_uniform_widths(orc):
    ms, mr, R = _stats(128, 8)
    w, off = orc.alloc(_cfg(orc, UNIFORM), ms, mr, R)
    assert np.all(w == 4)
    assert np.array_equal(off, np.arange(4) * 32 * 4 * 32 // 8)


def test_head_unit_has_no_range(orc):
    cfg = orc.Cfg(B=1, H=16, dk=128, dv=128, unit_kind=1, decay_kind=1, bbar_num=4, bmin=2,
                  bmax=16, weight_kind=RANGE)
    ms, mr, R = _stats(16, 9)
    assert np.all(orc.weights(cfg, ms, mr, R) == 1.0)


def test_invalid_weight_kind(orc):
    ms, mr, R = _stats(128, 10)
    with pytest.raises(ValueError):
        orc.weights(_cfg(orc, 9), ms, mr, R)
