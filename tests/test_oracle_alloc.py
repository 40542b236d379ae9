"""Pins of the oracle's allocation (Sec. 3, Eq. 3, Eq. 4 and the integer rounding after it)."""
import itertools
import math

import numpy as np
import pytest

from oracle import theory as th


def _proxy(c, b):
    return sum(float(ci) * 4.0 ** (-int(bi)) for ci, bi in zip(c, b))


def test_expm1_series_accuracy(orc):
    """The FP32 Taylor expm1 used by the weight is within 2 ulp of the true value on [0, 1]
    (where the erase statistic lives) and within 8 ulp up to 4 (after halvings)."""
    xs = np.concatenate([np.linspace(0, 4, 4001), np.logspace(-8, 0.6, 500)]).astype(np.float32)
    for x in xs:
        got = np.float32(orc.expm1_series(float(x)))
        ref = math.expm1(float(x))
        ulp = np.spacing(np.float32(ref)) if ref > 0 else np.float32(1e-45)
        tol = 2 if x <= 1 else 8
        assert abs(float(got) - ref) <= tol * float(ulp), (x, got, ref)
    assert orc.expm1_series(0.0) == 0.0


def test_weight_matches_eq3(orc):
    """FP32 weight from the EMAs equals Eq. (3) evaluated in FP64 (Rtilde = 1: equal ranges)."""
    rng = np.random.default_rng(0)
    cfg = orc.Cfg(B=1, H=2, dk=32, dv=32, group_heads=1, bbar_num=4, bmin=1, bmax=8)
    N = cfg.units
    s = np.exp(rng.uniform(np.log(1e-4), np.log(3.0), N))
    ms = (-np.expm1(-2 * s)).astype(np.float32)            # EMA of 1 - e^{-2s}
    mr = rng.uniform(0, 0.05, N).astype(np.float32)         # EMA of beta(2-beta)k^2
    R = np.ones(N, np.float32)
    c = orc.weights(cfg, ms, mr, R)
    ref = th.gamma_hat(th.s_hat_from_ema(1.0 - ms.astype(np.float64)), 0.5 * mr.astype(np.float64))
    assert np.allclose(c, ref, rtol=2e-5)


def test_weight_range_normalisation(orc):
    """Rtilde_i = R_i / RMS over the output-normalisation group (here 2 heads)."""
    rng = np.random.default_rng(1)
    cfg = orc.Cfg(B=1, H=4, dk=8, dv=8, group_heads=2, bbar_num=4, bmin=1, bmax=8)
    N = cfg.units
    ms = np.full(N, 0.5, np.float32)
    mr = np.zeros(N, np.float32)
    R = np.exp(rng.normal(0, 1, N)).astype(np.float32)
    c = orc.weights(cfg, ms, mr, R).astype(np.float64)
    G = 1.0  # (1 - 0.5) / (0 + 0.5)
    Rg = R.astype(np.float64).reshape(2, 16)
    ref = (G * Rg ** 2 / np.mean(Rg ** 2, axis=1, keepdims=True)).ravel()
    assert np.allclose(c, ref, rtol=1e-6)
    # all-zero group -> Rtilde = 1
    R0 = R.copy()
    R0[:16] = 0
    c0 = orc.weights(cfg, ms, mr, R0)
    assert np.allclose(c0[:16], 1.0)


@pytest.mark.parametrize("seed", range(6))
def test_integer_alloc_is_proxy_optimal_brute_force(orc, seed):
    """Budget met exactly, widths in range, and no other integer width vector with the same
    budget has a smaller high-rate proxy sum c_i 4^{-b_i} (enumerated, N <= 6)."""
    rng = np.random.default_rng(seed)
    N = int(rng.integers(2, 7))
    bmin, bmax = int(rng.integers(0, 3)), int(rng.integers(4, 9))
    bbar = int(rng.integers(bmin + 1, bmax))
    c = np.exp(rng.normal(0, 3, N)).astype(np.float32)
    w = orc.alloc_from_weights(c, bmin, bmax, N * bbar, bbar, 1)
    assert int(w.sum()) == N * bbar
    assert w.min() >= bmin and w.max() <= bmax
    best = min(_proxy(c, b) for b in itertools.product(range(bmin, bmax + 1), repeat=N)
               if sum(b) == N * bbar)
    assert _proxy(c, w) <= best * (1 + 1e-12)


def _literal_round_clip_adjust(c, bbar, bmin, bmax):
    """Sec. 3 read literally, in FP64: Eq. (4), round to nearest, clip, then move single bits
    by the rounding remainder b_real - b until the budget is met."""
    br = th.alloc_real(c, bbar)
    b = np.clip(np.floor(br + 0.5), bmin, bmax).astype(int)
    total = len(c) * bbar
    while b.sum() > total:
        key = np.where(b > bmin, br - b, np.inf)
        b[int(np.argmin(key))] -= 1
    while b.sum() < total:
        key = np.where(b < bmax, br - b, -np.inf)
        b[int(np.argmax(key))] += 1
    return b


@pytest.mark.parametrize("N,bbar,bmin,bmax,spread", [(64, 4, 0, 8, 2.0), (512, 2, 1, 8, 3.0),
                                                       (300, 6, 1, 16, 4.0), (128, 3, 1, 8, 0.3)])
def test_integer_alloc_equals_literal_procedure(orc, N, bbar, bmin, bmax, spread):
    rng = np.random.default_rng(N)
    c = np.exp(rng.normal(0, spread, N)).astype(np.float32)
    w = orc.alloc_from_weights(c, bmin, bmax, N * bbar, bbar, 1)
    ref = _literal_round_clip_adjust(c.astype(np.float64), bbar, bmin, bmax)
    assert np.array_equal(w.astype(int), ref)


def test_uniform_weights_give_uniform_widths(orc):
    for bbar in (1, 2, 4, 6):
        w = orc.alloc_from_weights(np.full(100, 0.37, np.float32), 0, 16, 100 * bbar, bbar, 1)
        assert np.all(w == bbar)
    # fractional mean: the extra bits go to the lowest indices
    w = orc.alloc_from_weights(np.ones(8, np.float32), 1, 8, 8 * 2 + 3, 19, 8)
    assert list(w) == [3, 3, 3, 2, 2, 2, 2, 2]


def test_head_unit_two_bit_floor_reduces_to_uniform_block(orc):
    """Sec. 3 'Allocation units': b_min = 2 with a two-bit mean gives every head 2 bits."""
    cfg = orc.Cfg(B=3, H=16, dk=128, dv=128, decay_kind=1, unit_kind=1, bbar_num=2, bmin=2,
                  bmax=16)
    rng = np.random.default_rng(5)
    ms = rng.uniform(0.001, 0.5, cfg.B * cfg.H).astype(np.float32)
    mr = rng.uniform(0, 0.01, cfg.B * cfg.H).astype(np.float32)
    widths, head_off = orc.alloc(cfg, ms, mr, np.zeros(cfg.B * cfg.H, np.float32))
    assert np.all(widths == 2)
    assert list(head_off[:3]) == [0, 2 * 128 * 128 // 8, 4 * 128 * 128 // 8]


def test_alloc_budget_offsets_and_infeasible(orc):
    rng = np.random.default_rng(6)
    cfg = orc.Cfg(B=4, H=3, dk=16, dv=16, group_heads=1, bbar_num=4, bmin=0, bmax=8)
    N = cfg.units
    ms = rng.uniform(1e-4, 0.9, cfg.B * N).astype(np.float32)
    mr = rng.uniform(0, 0.05, cfg.B * N).astype(np.float32)
    R = np.exp(rng.normal(0, 1, cfg.B * N)).astype(np.float32)
    widths, head_off = orc.alloc(cfg, ms, mr, R)
    wb = widths.reshape(cfg.B, cfg.H, cfg.dk).astype(int)
    assert np.all(wb.sum(axis=(1, 2)) == N * 4)
    row_bytes = wb * cfg.dv // 8
    exp_off = np.concatenate([np.zeros((cfg.B, 1), int),
                              np.cumsum(row_bytes.sum(axis=2), axis=1)[:, :-1]], axis=1)
    assert np.array_equal(head_off.reshape(cfg.B, cfg.H), exp_off)
    assert np.all(row_bytes.sum(axis=(1, 2)) == cfg.region_bytes)
    with pytest.raises(ValueError):
        orc.alloc_from_weights(np.ones(4, np.float32), 5, 8, 4 * 4, 4, 1)


def test_alloc_prefers_slow_rows_and_large_ranges(orc):
    """Widths grow with Gamma_hat (slow decay) and with the normalised range."""
    cfg = orc.Cfg(B=1, H=1, dk=64, dv=64, bbar_num=4, bmin=1, bmax=16)
    s = np.logspace(-3, 0, 64)
    ms = (-np.expm1(-2 * s)).astype(np.float32)
    w, _ = orc.alloc(cfg, ms, np.zeros(64, np.float32), np.ones(64, np.float32))
    assert np.all(np.diff(w.astype(int)) <= 0) and w[0] > w[-1]
    R = np.logspace(-1, 1, 64).astype(np.float32)
    w2, _ = orc.alloc(cfg, np.full(64, 0.1, np.float32), np.zeros(64, np.float32), R)
    assert np.all(np.diff(w2.astype(int)) >= 0) and w2[-1] > w2[0]
    # Eq. (4) spacing: a factor 4 in c is one bit when nothing clips (integer b_real here)
    c = (4.0 ** np.arange(5)).astype(np.float32)
    w3 = orc.alloc_from_weights(c, 0, 16, 5 * 8, 8, 1)
    assert list(w3) == [6, 7, 8, 9, 10]
    # exact ties at a rounding boundary (b_real = k + 5.5): lower index gets the bit
    c = (4.0 ** np.arange(6)).astype(np.float32)
    w4 = orc.alloc_from_weights(c, 0, 16, 6 * 8, 8, 1)
    assert list(w4) == [6, 7, 8, 8, 9, 10]
