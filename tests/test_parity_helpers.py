"""CPU pins of the parity helpers that the GPU tests rely on: the vectorised code decoder
against the oracle's own row decoder, on packed states of every width (row and head unit)."""
import numpy as np
import pytest

import synth
from parity import codes_fast, codes_of


def _packed_state(orc, w, lo, hi, seed):
    cfg = orc.Cfg.from_workload(w, bmin=lo, bmax=hi)
    rng = np.random.default_rng(seed)
    N = cfg.units
    total = N * cfg.bbar_num // cfg.bbar_den
    ws = []
    for _ in range(cfg.B):
        wv = np.full(N, total // N)
        for _ in range(6 * N):
            i, j = rng.integers(0, N, 2)
            if wv[i] < hi and wv[j] > lo:
                wv[i] += 1
                wv[j] -= 1
        ws.append(wv)
    widths = np.stack(ws).astype(np.uint8).ravel()
    rows = widths.reshape(cfg.B, -1)
    if cfg.unit_kind == 1:
        rows = np.repeat(rows, cfg.dk, axis=1)
    hb = (rows.reshape(cfg.B, cfg.H, cfg.dk).astype(int) * cfg.dv // 8).sum(2)
    head_off = np.concatenate([np.zeros((cfg.B, 1), int), np.cumsum(hb, 1)[:, :-1]], 1)
    S = synth.random_state(w, seed)
    payload, scales, fidx, _ = orc.pack(cfg, S, widths, head_off.astype(np.uint32).ravel())
    return cfg, orc.Buf(payload, scales, widths, head_off.astype(np.uint32).ravel(), fidx)


@pytest.mark.parametrize("name,lo,hi", [("kda_decode", 0, 16), ("mamba2_decode", 1, 16),
                                        ("gdn_decode", 2, 16), ("tiny_kda", 0, 8)])
def test_codes_fast_equals_oracle_row_decoder(orc, name, lo, hi):
    w = synth.scaled(synth.WORKLOADS[name], B=2, H=min(synth.WORKLOADS[name].H, 3), bmin=lo, bmax=hi)
    cfg, buf = _packed_state(orc, w, lo, hi, 5)
    c_ref, w_ref = codes_of(orc, cfg, buf)
    c_new, w_new = codes_fast(cfg, buf)
    assert np.array_equal(w_new, w_ref)
    assert np.array_equal(c_new, c_ref)
    assert len(np.unique(w_ref)) >= 3    # several widths in one state


def test_codes_fast_sees_a_flipped_bit(orc):
    w = synth.scaled(synth.WORKLOADS["kda_decode"], B=1, H=2)
    cfg, buf = _packed_state(orc, w, 1, 8, 9)
    c0, _ = codes_fast(cfg, buf)
    buf.payload[1000] ^= 0x10
    c1, _ = codes_fast(cfg, buf)
    c_ref, _ = codes_of(orc, cfg, buf)
    assert np.count_nonzero(c1 != c0) == 1
    assert np.array_equal(c1, c_ref)


def test_oracle_parallel_timing_build_is_the_same_computation(orc):
    """The OpenMP timing build of the oracle (heads of a write-back on several threads) gives
    the plain build's results bit for bit: readouts, packed state, statistics."""
    w = synth.scaled(synth.WORKLOADS["kda_decode"], B=2, H=6, T=3)
    cfg = orc.Cfg.from_workload(w)
    inp = synth.host_inputs(w)
    codes, lut, _ = orc.quant_decay(inp["s"], w.H * w.dk, w.gate_bits)
    outs = []
    for par in (False, True):
        src, dst = orc.init_state(cfg)
        ms, mr, R = (np.zeros(cfg.B * cfg.units, np.float32) for _ in range(3))
        o = np.zeros((w.B, w.T, w.H, w.dv), np.float32)
        for t in range(w.T):
            orc.step(cfg, src, dst, inp, t, t + 1, t, o, ms, mr, R, codes, lut, parallel=par)
            src.widths[:], src.head_off[:] = orc.alloc(cfg, ms, mr, R)
            src, dst = dst, src
        outs.append((o, src, ms, mr, R))
    (o0, s0, *st0), (o1, s1, *st1) = outs
    assert np.array_equal(o0.view(np.uint32), o1.view(np.uint32))
    for f in ("payload", "scales", "widths", "head_off", "fidx"):
        assert np.array_equal(getattr(s0, f), getattr(s1, f)), f
    for a, b in zip(st0, st1):
        assert np.array_equal(a.view(np.uint32), b.view(np.uint32))


def test_cand_step_is_the_oracles_stored_step(orc):
    from parity import cand_step
    rng = np.random.default_rng(3)
    for b in range(2, 12):
        for _ in range(20):
            x = (rng.standard_normal(64) * np.exp(rng.uniform(-8, 8))).astype(np.float32)
            _, scale, fidx = orc.quant_group(x, b)
            D = np.uint16(scale).view(np.float16).astype(np.float32)
            assert cand_step(fidx, np.max(np.abs(x)), b) == D


def test_range_samples_cover_every_step_pattern():
    from parity import cand_step, range_samples
    b = 4
    # a range whose candidate 15 (f = 1) sits right at an FP16 rounding boundary of R / 7
    mid = np.float32((np.float64(np.float16(0.5)) + np.float64(np.nextafter(np.float16(0.5), np.float16(1)))) / 2)
    R = np.float32(mid * np.float32(7.0))
    rs = range_samples(R, b, rel=1e-5)
    ulp = np.float64(np.spacing(R))
    assert all(abs(np.float64(r) - np.float64(R)) <= 1e-5 * np.float64(R) + ulp for r in rs)
    steps = {cand_step(15, r, b) for r in rs}
    assert len(steps) == 2                        # both sides of the boundary are sampled
    for a, z in zip(rs[:-1], rs[1:]):             # every step is constant between samples
        for k in range(16):
            m = np.float32((np.float64(a) + np.float64(z)) / 2)
            assert cand_step(k, m, b) in (cand_step(k, a, b), cand_step(k, z, b))


def test_factor_explained_by_range_accepts_the_oracles_choice_only(orc):
    from parity import cand_step, candidate_sse, factor_explained_by_range
    rng = np.random.default_rng(4)
    x = rng.standard_normal(128).astype(np.float32)
    b = 4
    _, scale, fidx = orc.quant_group(x, b)
    D = np.uint16(scale).view(np.float16).astype(np.float32)
    R = np.max(np.abs(x))
    assert factor_explained_by_range(x, b, fidx, D, R)
    sse = candidate_sse(x, b, R)
    worst = int(np.argmax(sse))
    assert not factor_explained_by_range(x, b, worst, cand_step(worst, R, b), R)


def test_rel_err_tokens_is_normwise_per_token():
    from parity import rel_err_tokens, rel_err_vectors
    ref = np.ones((2, 3, 4, 8), np.float32)
    ref[0, 1, 2] = 1e-6                            # a nearly cancelled readout
    a = ref.copy()
    a[0, 1, 2] += 1e-6                             # 100 % off for that vector
    assert rel_err_vectors(a, ref) > 0.5
    assert rel_err_tokens(a, ref) < 1e-6
    a[1, 2] += 1e-3
    assert abs(rel_err_tokens(a, ref) - 1e-3 / np.sqrt(2)) < 1e-4
