"""Pins of the oracle's recurrence (Eq. 1) and of its write-back step (Sec. 2 "Accumulated
readout error", Sec. 3 statistics, Sec. 5 protocol)."""
import numpy as np
import pytest

import synth


def _unit(rng, *shape):
    g = rng.standard_normal(shape)
    return g / np.linalg.norm(g, axis=-1, keepdims=True)


def test_delta_rule_writes_value_exactly(orc):
    """KDA/GDN with beta = 1 and a unit key: after the update S_t^T k_t = v_t (the delta rule
    replaces the value stored under k_t)."""
    rng = np.random.default_rng(0)
    dk, dv, T = 16, 8, 30
    k = _unit(rng, T, dk).astype(np.float32)
    k = (k / np.linalg.norm(k.astype(np.float64), axis=1, keepdims=True)).astype(np.float32)
    q = _unit(rng, T, dk).astype(np.float32)
    v = rng.standard_normal((T, dv)).astype(np.float32)
    s = rng.uniform(0, 0.5, (T, dk)).astype(np.float32)
    S = rng.standard_normal((dk, dv))
    for t in range(T):
        _, S = orc.recur(S, k[t:t + 1], q[t:t + 1], v[t:t + 1], s[t:t + 1], k[t:t + 1],
                         np.ones((1, dv), np.float32), dtype=np.float64)
        kt = k[t].astype(np.float64)
        assert np.allclose(S.T @ kt, v[t] * (kt @ kt), atol=1e-12)


def test_no_erase_closed_form(orc):
    """Mamba-2 form (a = 0, w = 1), constant per-head decay: one write k0 v0^T then zero
    writes gives o_t = e^{-s t} (k0 . q_t) v0."""
    rng = np.random.default_rng(1)
    dk, dv, T, s0 = 8, 4, 40, 0.07
    k = np.zeros((T, dk), np.float32)
    k[0] = rng.standard_normal(dk)
    q = rng.standard_normal((T, dk)).astype(np.float32)
    v = np.zeros((T, dv), np.float32)
    v[0] = rng.standard_normal(dv)
    s = np.full((T, dk), s0, np.float32)
    o, _ = orc.recur(np.zeros((dk, dv)), k, q, v, s, np.zeros_like(k),
                     np.ones((T, dv), np.float32), dtype=np.float64)
    t = np.arange(T)[:, None]
    ref = np.exp(-np.float64(np.float32(s0)) * t) * (q.astype(np.float64) @ k[0].astype(np.float64))[:, None] * v[0]
    assert np.allclose(o, ref, rtol=1e-12, atol=1e-14)


def test_delta_form_equals_general_form(orc):
    """Eq. (1) with a = beta k, w = beta 1 equals S' + beta k (v - S'^T k)^T (restated in FP64
    numpy), with o read from the updated state."""
    rng = np.random.default_rng(2)
    dk, dv, T = 12, 6, 25
    k = _unit(rng, T, dk).astype(np.float32)
    q = _unit(rng, T, dk).astype(np.float32)
    v = rng.standard_normal((T, dv)).astype(np.float32)
    s = rng.uniform(0.001, 1.0, (T, dk)).astype(np.float32)
    beta = rng.choice([0.125, 0.25, 0.5, 1.0], T).astype(np.float32)   # beta k exact in FP32
    S0 = rng.standard_normal((dk, dv))
    o, ST = orc.recur(S0, k, q, v, s, (beta[:, None] * k).astype(np.float32),
                      np.repeat(beta[:, None], dv, 1).astype(np.float32), dtype=np.float64)
    S = S0.copy()
    for t in range(T):
        kt, qt = k[t].astype(np.float64), q[t].astype(np.float64)
        bt = np.float64(beta[t])
        Sp = np.exp(-s[t].astype(np.float64))[:, None] * S
        S = Sp + bt * np.outer(kt, v[t] - Sp.T @ kt)
        assert np.allclose(o[t], S.T @ qt, rtol=1e-12, atol=1e-12)
    assert np.allclose(ST, S, rtol=1e-12, atol=1e-12)


def test_fp32_tracks_fp64(orc):
    w = synth.WORKLOADS["tiny_kda"]
    inp = synth.host_inputs(w)
    cfg = orc.Cfg.from_workload(w)
    args = orc.expand_inputs(cfg, inp, 0, 0)
    o32, _ = orc.recur(np.zeros((w.dk, w.dv)), *args, dtype=np.float32)
    o64, _ = orc.recur(np.zeros((w.dk, w.dv)), *args, dtype=np.float64)
    rel = np.linalg.norm(o32 - o64, axis=1) / np.maximum(np.linalg.norm(o64, axis=1), 1e-30)
    assert rel.max() < 1e-5


# --------------------------------- write-back step / scan ---------------------------------
def _small(name, **kw):
    base = synth.WORKLOADS[name]
    return synth.scaled(base, **kw)


@pytest.mark.parametrize("name,kw", [
    ("tiny_kda", dict(T=40)),
    ("kda_decode", dict(B=2, H=2, dk=32, dv=32, T=12, gate_bits=0)),
    ("gdn_decode", dict(B=2, H=3, dk=64, dv=32, T=10)),
    ("mamba2_decode", dict(B=2, H=4, dk=32, dv=16, T=10, group_heads=2)),
    ("kda_prefill", dict(B=1, H=2, dk=32, dv=32, T=70, C=16)),
])
def test_scan_budget_and_lagged_widths(orc, name, kw):
    """Every write-back meets the layer budget exactly, widths stay in range, and the widths
    used at write-back w+1 are the allocation of the statistics left by write-back w."""
    w = _small(name, **kw)
    cfg = orc.Cfg.from_workload(w)
    inp = synth.host_inputs(w)
    src, dst = orc.init_state(cfg)
    o = np.zeros((w.B, w.T, w.H, w.dv), np.float32)
    ms, mr, R = (np.zeros(cfg.B * cfg.units, np.float32) for _ in range(3))
    for wi, t0 in enumerate(range(0, w.T, w.C)):
        t1 = min(w.T, t0 + w.C)
        orc.step(cfg, src, dst, inp, t0, t1, wi, o, ms, mr, R)
        nw, no = orc.alloc(cfg, ms, mr, R)
        wb = nw.reshape(cfg.B, -1).astype(int)
        per = wb if cfg.unit_kind == 0 else wb
        assert np.all(per.sum(1) == cfg.units * w.bbar)
        assert nw.min() >= w.bmin and nw.max() <= w.bmax
        src.widths[:], src.head_off[:] = nw, no
        src, dst = dst, src
    assert np.all(np.isfinite(o))


def test_inconsistent_layout_is_rejected(orc):
    """Widths beyond 16 or offsets running past the region are refused, not written."""
    w = _small("kda_decode", B=1, H=2, dk=32, dv=32, T=1, gate_bits=0)
    cfg = orc.Cfg.from_workload(w)
    src, dst = orc.init_state(cfg)
    bad = dst.copy()
    bad.widths[0] = 200
    o = np.zeros((1, 1, w.H, w.dv), np.float32)
    z = np.zeros(cfg.units, np.float32)
    with pytest.raises(ValueError):
        orc.step(cfg, src, bad, synth.host_inputs(w), 0, 1, 0, o, z, z.copy(), z.copy())
    bad = dst.copy()
    bad.head_off[1] = cfg.region_bytes - 8
    with pytest.raises(ValueError):
        orc.unpack(cfg, src.payload, src.scales, bad.widths, bad.head_off)


def test_outputs_precede_quantisation(orc):
    """o_t is read from the FP32 state before the write-back: changing the target widths
    (or the quantiser altogether) leaves every readout of the interval unchanged, and the
    readouts equal the plain FP32 recurrence from the dequantised state."""
    w = _small("kda_prefill", B=1, H=2, dk=32, dv=32, T=8, C=8)
    cfg = orc.Cfg.from_workload(w)
    inp = synth.host_inputs(w)
    rng = np.random.default_rng(3)
    S = synth.random_state(w, 2)
    src, dst = orc.init_state(cfg)
    src.payload[:], src.scales[:], src.fidx[:], _ = orc.pack(cfg, S, src.widths, src.head_off)
    outs = []
    for trial in range(2):
        d = dst.copy()
        if trial:
            pool = np.tile(np.array([1, 5, 2, 4, 3, 3]), 11)[:cfg.units]   # mean exactly 3
            assert pool.sum() == cfg.units * w.bbar
            d.widths[:] = np.tile(pool, cfg.B)
            rb = pool.reshape(w.H, w.dk).sum(1) * w.dv // 8
            d.head_off[:] = np.concatenate([[0], np.cumsum(rb)[:-1]])
        o = np.zeros((w.B, w.T, w.H, w.dv), np.float32)
        z = np.zeros(cfg.B * cfg.units, np.float32)
        orc.step(cfg, src, d, inp, 0, w.T, 0, o, z.copy(), z.copy(), z.copy())
        outs.append(o)
    assert np.array_equal(outs[0], outs[1])
    X0 = orc.unpack(cfg, src.payload, src.scales, src.widths, src.head_off)
    for h in range(w.H):
        ref, _ = orc.recur(X0[0, h], *orc.expand_inputs(cfg, inp, 0, h), dtype=np.float64)
        rel = np.linalg.norm(outs[0][0, :, h] - ref) / np.linalg.norm(ref)
        assert rel < 1e-5


def test_sixteen_bit_state_tracks_fp32(orc):
    """With every width at 16 bits the quantised scan follows the unquantised recurrence; the
    residual error comes from the FP16 scale (Delta = FP16(f R / n) may round below R / n, so
    the row maximum clips by up to 2^-11 R per write-back), far below the 2-bit error."""
    w = _small("tiny_kda", T=64, bbar=16, bmin=16, bmax=16)
    cfg = orc.Cfg.from_workload(w)
    inp = synth.host_inputs(w)
    o, *_ = orc.scan(cfg, inp)
    ref, _ = orc.recur(np.zeros((w.dk, w.dv)), *orc.expand_inputs(cfg, inp, 0, 0),
                       dtype=np.float64)
    rel = np.linalg.norm(o[0, :, 0] - ref, axis=1) / np.linalg.norm(ref, axis=1)
    assert rel.max() < 5e-3
    w2 = _small("tiny_kda", T=64)
    o2, *_ = orc.scan(orc.Cfg.from_workload(w2), inp)
    rel2 = np.linalg.norm(o2[0, :, 0] - ref, axis=1) / np.linalg.norm(ref, axis=1)
    assert rel2.mean() > 20 * rel.mean()


def test_ema_statistics_closed_form(orc):
    """EMA of span 64 per token: m_T = (1-a)^{T-1} x_0 + sum_{t>=1} a (1-a)^{T-1-t} x_t, with
    x_s = 1 - e^{-2 s} and x_r = beta (2 - beta) k_i^2 (row unit); and R_i is the row absmax
    of the state before quantisation."""
    w = _small("kda_prefill", B=1, H=1, dk=16, dv=16, T=50, C=50)
    cfg = orc.Cfg.from_workload(w)
    inp = synth.host_inputs(w)
    src, dst = orc.init_state(cfg)
    o = np.zeros((w.B, w.T, w.H, w.dv), np.float32)
    ms, mr, R = (np.zeros(cfg.units, np.float32) for _ in range(3))
    X = orc.step(cfg, src, dst, inp, 0, w.T, 0, o, ms, mr, R, want_x=True)
    a = 2.0 / 65.0
    s = inp["s"][0, :, 0].astype(np.float64)
    beta = inp["beta"][0, :, 0].astype(np.float64)
    k = inp["k"][0, :, 0].astype(np.float64)
    wts = np.array([(1 - a) ** (w.T - 1)] + [a * (1 - a) ** (w.T - 1 - t) for t in range(1, w.T)])
    ref_s = wts @ (-np.expm1(-2 * s))
    ref_r = wts @ (beta[:, None] * (2 - beta[:, None]) * k ** 2)
    assert np.allclose(ms, ref_s, rtol=2e-5)
    assert np.allclose(mr, ref_r, rtol=2e-5)
    assert np.array_equal(R, np.max(np.abs(X[0, 0]), axis=1))


def test_fit_every_reuses_factor(orc):
    """fit_every = K: heads refit when (w + h) % K == 0 and otherwise keep the stored factor."""
    w = _small("kda_decode", B=1, H=4, dk=32, dv=32, T=6, gate_bits=0)
    cfg = orc.Cfg.from_workload(w, fit_every=4)
    inp = synth.host_inputs(w)
    src, dst = orc.init_state(cfg)
    o = np.zeros((w.B, w.T, w.H, w.dv), np.float32)
    ms, mr, R = (np.zeros(cfg.units, np.float32) for _ in range(3))
    prev = src.fidx.copy()
    for wi in range(w.T):
        orc.step(cfg, src, dst, inp, wi, wi + 1, wi, o, ms, mr, R)
        cur = dst.fidx.reshape(w.H, w.dk)
        for h in range(w.H):
            if (wi + h) % 4 != 0:
                assert np.array_equal(cur[h], prev.reshape(w.H, w.dk)[h])
        prev = dst.fidx.copy()
        src.widths[:], src.head_off[:] = orc.alloc(cfg, ms, mr, R)
        src, dst = dst, src


def test_chunked_ragged_tail_matches_token_loop_without_quantisation_error(orc):
    """C > 1 with a ragged last chunk runs; the first chunk's readouts equal the FP32
    recurrence from the zero state (nothing has been quantised yet)."""
    w = _small("kda_prefill", B=1, H=1, dk=32, dv=32, T=37, C=16)
    cfg = orc.Cfg.from_workload(w)
    inp = synth.host_inputs(w)
    o, buf, *_ = orc.scan(cfg, inp)
    ref, _ = orc.recur(np.zeros((w.dk, w.dv), np.float32), *orc.expand_inputs(cfg, inp, 0, 0))
    assert np.array_equal(o[0, :16, 0], ref[:16])
    assert np.all(np.isfinite(o))


def _general_from_delta(inp):
    """General-erasure inputs that reproduce the delta rule: a = fl(beta k), w = beta 1."""
    g = dict(inp)
    g["a"] = (inp["beta"][..., None] * inp["k"]).astype(np.float32)
    g["w"] = np.repeat(inp["beta"][..., None], inp["v"].shape[-1], axis=-1).astype(np.float32)
    return g


def test_general_erasure_reproduces_delta_rule(orc):
    """With a = beta k and w = beta 1 the general form of Eq. (1) is the delta rule: the same
    readouts and packed state bit for bit; its erasure statistic 2 a_i k_i - a_i^2 |k|^2 is
    beta (2 - beta) k_i^2 up to rounding for unit keys."""
    w = _small("kda_decode", B=2, H=3, T=6)
    inp = synth.host_inputs(w)
    gin = _general_from_delta(inp)
    res = {}
    for kind, data in ((0, inp), (2, gin)):
        cfg = orc.Cfg.from_workload(w, erase_kind=kind, gate_bits=0)
        src, dst = orc.init_state(cfg)
        o = np.zeros((w.B, w.T, w.H, w.dv), np.float32)
        ms, mr, R = (np.zeros(cfg.B * cfg.units, np.float32) for _ in range(3))
        for t in range(w.T):
            orc.step(cfg, src, dst, data, t, t + 1, t, o, ms, mr, R)
            src.widths[:], src.head_off[:] = orc.alloc(cfg, ms, mr, R) if t == 0 else (dst.widths, dst.head_off)
            src, dst = dst, src
        res[kind] = (o.copy(), src.payload.copy(), ms.copy(), mr.copy())
    assert np.array_equal(res[0][0], res[2][0])
    assert np.array_equal(res[0][1], res[2][1])
    assert np.array_equal(res[0][2], res[2][2])
    assert np.allclose(res[0][3], res[2][3], rtol=2e-6, atol=1e-9)


def test_general_erasure_step_matches_recurrence(orc):
    """The quantised scan with general a and w at 16 bits follows the unquantised general
    recurrence (a second, independent implementation of Eq. (1) in the oracle)."""
    w = synth.scaled(synth.EXTENSION_WORKLOADS["kda_general"], B=1, H=1, dk=64, dv=64, T=40,
                     bbar=16, bmin=16, bmax=16)
    cfg = orc.Cfg.from_workload(w)
    assert cfg.erase_kind == 2
    inp = synth.host_inputs(w)
    o, *_ = orc.scan(cfg, inp)
    ref, _ = orc.recur(np.zeros((w.dk, w.dv)), *orc.expand_inputs(cfg, inp, 0, 0), dtype=np.float64)
    rel = np.linalg.norm(o[0, :, 0] - ref, axis=1) / np.linalg.norm(ref, axis=1)
    assert rel.max() < 5e-3
    # and it is not the delta rule: the perturbed a and the write gates change the readouts
    dref, _ = orc.recur(np.zeros((w.dk, w.dv)),
                        *orc.expand_inputs(orc.Cfg.from_workload(w, erase_kind=0), inp, 0, 0),
                        dtype=np.float64)
    assert np.linalg.norm(ref - dref) > 0.1 * np.linalg.norm(ref)


def test_general_erasure_needs_a_and_w(orc):
    w = _small("kda_decode", B=1, H=1, T=2)
    cfg = orc.Cfg.from_workload(w, erase_kind=2, gate_bits=0)
    src, dst = orc.init_state(cfg)
    o = np.zeros((1, w.T, 1, w.dv), np.float32)
    z = lambda: np.zeros(cfg.B * cfg.units, np.float32)
    with pytest.raises(ValueError):
        orc.step(cfg, src, dst, synth.host_inputs(w), 0, 1, 0, o, z(), z(), z())


def test_current_allocation_uses_this_write_backs_statistics(orc):
    """alloc_mode 1: the widths a write-back packs with are the allocation of the statistics
    that write-back produced (its own ranges and EMAs), and the budget still holds; with
    alloc_mode 0 they are those of the previous write-back."""
    w = _small("kda_decode", B=2, H=3, T=5, gate_bits=0)
    for mode in (0, 1):
        cfg = orc.Cfg.from_workload(w, alloc_mode=mode)
        inp = synth.host_inputs(w)
        src, dst = orc.init_state(cfg)
        o = np.zeros((w.B, w.T, w.H, w.dv), np.float32)
        ms, mr, R = (np.zeros(cfg.B * cfg.units, np.float32) for _ in range(3))
        for t in range(w.T):
            before = orc.alloc(cfg, ms, mr, R)[0] if t else None
            orc.step(cfg, src, dst, inp, t, t + 1, t, o, ms, mr, R)
            now = orc.alloc(cfg, ms, mr, R)[0]
            if mode == 1:
                assert np.array_equal(dst.widths, now)
            elif t:
                assert np.array_equal(dst.widths, before)
            assert dst.widths.reshape(w.B, -1).sum(axis=1).tolist() == [cfg.units * 4] * w.B
            if mode == 0:
                src.widths[:], src.head_off[:] = orc.alloc(cfg, ms, mr, R)
            src, dst = dst, src


def test_current_allocation_tracks_ranges_better_at_low_bits(orc):
    """Widths from the current ranges follow the state being quantised; on a two-bit budget
    they give a readout error no worse than lagged widths over a short scan."""
    w = _small("tiny_kda", T=96, bbar=2, bmin=1, bmax=8)
    inp = synth.host_inputs(w)
    ref, _ = orc.recur(np.zeros((w.dk, w.dv)), *orc.expand_inputs(orc.Cfg.from_workload(w), inp, 0, 0),
                       dtype=np.float64)
    err = {}
    for mode in (0, 1):
        o, *_ = orc.scan(orc.Cfg.from_workload(w, alloc_mode=mode), inp)
        err[mode] = float(np.mean((o[0, :, 0] - ref) ** 2) / np.mean(ref ** 2))
    assert err[1] <= 1.05 * err[0], err
