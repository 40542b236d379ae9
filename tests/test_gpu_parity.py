"""GPU parity tests: the CUDA library (through the C ABI) against the CPU oracle on identical
seeded inputs.  Bit-exact: allocation, initial state, pack/unpack layout, log-decay codes.
Floating point: unquantised FP32 recurrence (free-running, 1e-5), quantised write-backs in
lockstep (the oracle's state at each write-back is handed to the GPU; codes >= 99.99%
identical and within one step, readouts within 1e-5: they precede quantisation, so from the
same packed state they differ by FP32 rounding only)."""
import numpy as np
import pytest

import synth
from concurrent.futures import ThreadPoolExecutor

from parity import (REL_O_FP32, REL_O_LOCKSTEP, REL_O_QUANT, REL_STATS, compare_packed, dev,
                    from_gpu_state, host, rel_err_tokens, rel_err_vectors, set_gpu_state)

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")


def small(name, **kw):
    return synth.scaled(synth.WORKLOADS[name], **kw)


SMALL = {
    "tiny_kda": small("tiny_kda", T=48),
    "kda_decode": small("kda_decode", B=3, H=4, T=12),
    "gdn_decode": small("gdn_decode", B=3, H=5, T=10),
    "mamba2_decode": small("mamba2_decode", B=2, H=16, T=10, group_heads=8),
    "kda_prefill": small("kda_prefill", B=2, H=3, T=150, C=64),
}


def _dev_inputs(w, inp, q, s_code=None, s_lut=None):
    d = {k: dev(v, torch) for k, v in inp.items()}
    a, wg = d.get("a"), d.get("w")
    if s_code is not None:
        return q.Inputs(d["q"], d["k"], d["v"], None, dev(s_code, torch), dev(s_lut, torch),
                        d["beta"], w.T, a, wg), d
    return q.Inputs(d["q"], d["k"], d["v"], d["s"], None, None, d["beta"], w.T, a, wg), d


def _random_stats(cfg, rng, zero_group=False, null_rows=0):
    n = cfg.B * cfg.units
    s = np.exp(rng.uniform(np.log(1e-4), np.log(3.0), n))
    ms = (-np.expm1(-2 * s)).astype(np.float32)
    mr = rng.uniform(0, 0.05, n).astype(np.float32)
    R = np.exp(rng.normal(0, 1.5, n)).astype(np.float32)
    if zero_group:
        R[: cfg.group_heads * cfg.dk] = 0
    if null_rows:
        ms[rng.choice(n, null_rows, replace=False)] = 1.0   # Gamma_hat = 0
    return ms, mr, R


# ------------------------------------------------------------------------------ bit-exact units
@pytest.mark.parametrize("name", ["tiny_kda", "kda_decode", "gdn_decode", "mamba2_decode", "kda_prefill"])
def test_alloc_bit_exact(qs, orc, name):
    w = synth.WORKLOADS[name]
    w = synth.scaled(w, B=min(w.B, 6))
    cfgq, cfgo = qs.Config.from_workload(w), orc.Cfg.from_workload(w)
    rng = np.random.default_rng(7)
    for trial in range(4):
        ms, mr, R = _random_stats(cfgo, rng, zero_group=(trial == 1), null_rows=7 if trial == 2 else 0)
        if trial == 3:
            ms[:] = ms[0]; mr[:] = mr[0]; R[:] = R[0]           # all tied
        st = qs.Stats(dev(ms, torch), dev(mr, torch), dev(R, torch))
        widths = torch.zeros(cfgq.B * cfgq.units, dtype=torch.uint8, device="cuda")
        head_off = torch.zeros(cfgq.B * cfgq.H, dtype=torch.int32, device="cuda")
        qs.qstate_alloc_bits(cfgq, st, widths, head_off)
        qs.qstate_check()
        wref, oref = orc.alloc(cfgo, ms, mr, R)
        assert np.array_equal(host(widths, np.uint8), wref), (name, trial)
        assert np.array_equal(host(head_off, np.uint32), oref), (name, trial)


@pytest.mark.parametrize("kind", range(9))
@pytest.mark.parametrize("name", ["kda_decode", "gdn_decode", "mamba2_decode"])
def test_alloc_weight_kinds_bit_exact(qs, orc, name, kind):
    """The allocation weights of Table 1 (weight_kind 1-8) give the oracle's widths bit for bit."""
    w = synth.scaled(synth.WORKLOADS[name], B=3)
    over = dict(weight_kind=kind, C=16 if kind == 5 else w.C)
    cfgq, cfgo = qs.Config.from_workload(w, **over), orc.Cfg.from_workload(w, **over)
    rng = np.random.default_rng(100 + kind)
    ms, mr, R = _random_stats(cfgo, rng, null_rows=3)
    st = qs.Stats(dev(ms, torch), dev(mr, torch), dev(R, torch))
    widths = torch.zeros(cfgq.B * cfgq.units, dtype=torch.uint8, device="cuda")
    head_off = torch.zeros(cfgq.B * cfgq.H, dtype=torch.int32, device="cuda")
    qs.qstate_alloc_bits(cfgq, st, widths, head_off)
    qs.qstate_check()
    wref, oref = orc.alloc(cfgo, ms, mr, R)
    assert np.array_equal(host(widths, np.uint8), wref)
    assert np.array_equal(host(head_off, np.uint32), oref)


@pytest.mark.parametrize("name", ["tiny_kda", "kda_decode", "gdn_decode", "mamba2_decode"])
def test_init_bit_exact(qs, orc, name):
    w = synth.scaled(synth.WORKLOADS[name], B=2)
    cfgq, cfgo = qs.Config.from_workload(w), orc.Cfg.from_workload(w)
    a, b = qs.new_state(cfgq), qs.new_state(cfgq)
    qs.qstate_init(cfgq, a, b)
    qs.qstate_check()
    ra, rb = orc.init_state(cfgo)
    ga, gb = from_gpu_state(orc, a), from_gpu_state(orc, b)
    for f in ("payload", "scales", "widths", "head_off", "fidx"):
        assert np.array_equal(getattr(ga, f), getattr(ra, f)), f
    assert np.array_equal(gb.widths, rb.widths) and np.array_equal(gb.head_off, rb.head_off)


def _width_map(cfgo, rng, lo, hi):
    """Random widths in [lo, hi] meeting the budget exactly, with offsets."""
    N = cfgo.units
    total = N * cfgo.bbar_num // cfgo.bbar_den
    ws = []
    for b in range(cfgo.B):
        w = np.full(N, total // N)
        for _ in range(4 * N):
            i, j = rng.integers(0, N, 2)
            if w[i] < hi and w[j] > lo:
                w[i] += 1
                w[j] -= 1
        ws.append(w)
    wv = np.stack(ws).astype(np.uint8)
    rows = wv if cfgo.unit_kind == 0 else np.repeat(wv, cfgo.dk, axis=1)
    row_bytes = rows.reshape(cfgo.B, cfgo.H, cfgo.dk).astype(int) * cfgo.dv // 8
    hb = row_bytes.sum(2)
    off = np.concatenate([np.zeros((cfgo.B, 1), int), np.cumsum(hb, 1)[:, :-1]], 1)
    return wv.ravel(), off.astype(np.uint32).ravel()


@pytest.mark.parametrize("name,lo,hi", [("kda_decode", 0, 16), ("tiny_kda", 0, 16),
                                        ("gdn_decode", 2, 16), ("mamba2_decode", 1, 16)])
def test_pack_unpack_vs_oracle(qs, orc, name, lo, hi):
    _pack_unpack(qs, orc, synth.scaled(synth.WORKLOADS[name], B=2, bmin=lo, bmax=hi), lo, hi)


# Head unit at the other supported state shapes: 128 x 64 takes the kernel whose lanes own one
# whole scale group each (one value column per lane there), 64 x 64 the general kernel.
HEAD_SHAPES = [(128, 64), (64, 64)]


@pytest.mark.parametrize("dk,dv", HEAD_SHAPES)
def test_pack_unpack_head_unit_shapes(qs, orc, dk, dv):
    _pack_unpack(qs, orc, synth.scaled(synth.WORKLOADS["gdn_decode"], B=2, H=3, dk=dk, dv=dv), 0, 16)


def _pack_unpack(qs, orc, w, lo, hi):
    cfgq, cfgo = qs.Config.from_workload(w), orc.Cfg.from_workload(w)
    rng = np.random.default_rng(11)
    widths, head_off = _width_map(cfgo, rng, lo, hi)
    S = synth.random_state(w, 3)
    # edge rows: all zero, a single spike, tiny (FP16 subnormal steps) and huge ranges
    S[0, 0, 0] = 0
    S[0, 0, 1] = 0
    S[0, 0, 1, 5] = -3.0
    S[0, 0, 2] *= 1e-6
    S[0, 0, 3] *= 1e3
    ref_payload, ref_scales, ref_fidx, ref_range = orc.pack(cfgo, S, widths, head_off)
    ref = orc.Buf(ref_payload, ref_scales, widths, head_off, ref_fidx)
    st = qs.new_state(cfgq)
    st.widths.copy_(dev(widths, torch))
    st.head_off.copy_(dev(head_off, torch))
    rng_out = torch.zeros(cfgq.B * cfgq.units, dtype=torch.float32, device="cuda")
    qs.qstate_pack(cfgq, dev(S, torch), st, rng_out if cfgq.unit_kind == 0 else None)
    qs.qstate_check()
    gpu = from_gpu_state(orc, st)
    compare_packed(orc, cfgo, gpu, ref, X=S)
    if cfgq.unit_kind == 0:
        assert np.array_equal(host(rng_out, np.float32), ref_range)
    # unpack is bit-exact on both payloads
    for buf in (ref, gpu):
        set_gpu_state(st, buf)
        out = torch.empty(S.shape, dtype=torch.float32, device="cuda")
        qs.qstate_unpack(cfgq, st, out)
        qs.qstate_check()
        X = orc.unpack(cfgo, buf.payload, buf.scales, buf.widths, buf.head_off)
        assert np.array_equal(host(out, np.float32), X)


@pytest.mark.parametrize("name,g", [("kda_decode", 2), ("kda_decode", 4), ("gdn_decode", 2),
                                    ("mamba2_decode", 1)])
def test_quant_decay_bit_exact(qs, orc, name, g):
    w = synth.scaled(synth.WORKLOADS[name], B=3, T=40, gate_bits=g)
    cfgq = qs.Config.from_workload(w)
    inp = synth.host_inputs(w)
    s = inp["s"]
    nchan = w.H * w.dk if w.per_row_decay else w.H
    codes = torch.zeros(s.shape, dtype=torch.uint8, device="cuda")
    lut = torch.zeros(nchan * 2 ** g, dtype=torch.float32, device="cuda")
    thr = torch.zeros(nchan * (2 ** g - 1), dtype=torch.float32, device="cuda")
    qs.qstate_quant_decay(cfgq, dev(s, torch), codes, lut, thr)
    qs.qstate_check()
    c_ref, l_ref, t_ref = orc.quant_decay(s, nchan, g)
    assert np.array_equal(host(lut, np.float32).reshape(nchan, -1), l_ref)
    assert np.array_equal(host(thr, np.float32).reshape(nchan, -1), t_ref)
    assert np.array_equal(host(codes, np.uint8), c_ref)


# ------------------------------------------------------------------ unquantised FP32 recurrence
@pytest.mark.parametrize("name", ["tiny_kda", "kda_decode", "gdn_decode", "mamba2_decode", "kda_prefill"])
def test_fp32_recurrence_free_running(qs, orc, name):
    w = SMALL[name] if name != "tiny_kda" else synth.WORKLOADS["tiny_kda"]
    cfgq, cfgo = qs.Config.from_workload(w, gate_bits=0), orc.Cfg.from_workload(w, gate_bits=0)
    inp = synth.host_inputs(w)
    X, _ = _dev_inputs(w, inp, qs)
    S = torch.zeros((w.B, w.H, w.dk, w.dv), dtype=torch.float32, device="cuda")
    o = torch.zeros((w.B, w.T, w.H, w.dv), dtype=torch.float32, device="cuda")
    qs.qstate_scan_fp32(cfgq, S, X, 0, w.T, o)
    qs.qstate_check()
    og = host(o, np.float32)
    worst32 = worst64 = 0.0
    for b in range(w.B):
        for h in range(w.H):
            args = orc.expand_inputs(cfgo, inp, b, h)
            o32, _ = orc.recur(np.zeros((w.dk, w.dv)), *args, dtype=np.float32)
            o64, _ = orc.recur(np.zeros((w.dk, w.dv)), *args, dtype=np.float64)
            worst32 = max(worst32, rel_err_vectors(og[b, :, h], o32))
            worst64 = max(worst64, rel_err_vectors(og[b, :, h], o64))
    print(f"{name}: max rel readout error vs FP32 oracle {worst32:.2e}, vs FP64 {worst64:.2e}")
    assert worst32 <= REL_O_FP32
    assert worst64 <= REL_O_FP32


# --------------------------------------------------------------- quantised write-backs, lockstep
def _lockstep(qs, orc, w, fit_every=1, log_decay=False, sample_b=None, max_wb=None, weight_kind=0,
              interval_form=0, inputs=None, oracle_parallel=False):
    """Run the oracle free; before every write-back copy its state into the GPU, run one
    qstate_step and compare the GPU's write-back with the oracle's.  With sample_b, the GPU
    runs the full batch and only those batch elements are injected and compared (the oracle
    runs a B=1 configuration per sampled element, one host thread each).  interval_form
    selects the library's token-by-token or chunked computation of each interval (the oracle
    is always token by token).  Returns the per-write-back report and the oracle's
    free-running readouts per compared element.  oracle_parallel runs the oracle's OpenMP
    build (the heads of a write-back on several threads; the same results bit for bit, pinned
    on the CPU)."""
    cfgq = qs.Config.from_workload(w, fit_every=fit_every, weight_kind=weight_kind,
                                   interval_form=interval_form)
    cfgo_full = orc.Cfg.from_workload(w, fit_every=fit_every, weight_kind=weight_kind)
    inp = synth.host_inputs(w) if inputs is None else inputs
    s_code = s_lut = None
    if log_decay:
        nchan = w.H * w.dk if w.per_row_decay else w.H
        s_code, s_lut, _ = orc.quant_decay(inp["s"], nchan, w.gate_bits)
    X, _ = _dev_inputs(w, inp, qs, s_code, s_lut)
    bs = list(range(w.B)) if sample_b is None else list(sample_b)
    one = sample_b is not None
    cfgo = (orc.Cfg.from_workload(synth.scaled(w, B=1), fit_every=fit_every, weight_kind=weight_kind)
            if one else cfgo_full)
    sub = (lambda a, b: a[b:b + 1]) if one else (lambda a, b: a)
    orc_inp = {b: {k: sub(v, b) for k, v in inp.items()} for b in (bs if one else [0])}
    orc_code = {b: (sub(s_code, b) if s_code is not None else None) for b in (bs if one else [0])}
    # oracle states per (sampled) batch element
    states = {}
    for key in (bs if one else [0]):
        src, dst = orc.init_state(cfgo)
        z = lambda: np.zeros(cfgo.B * cfgo.units, np.float32)
        states[key] = dict(src=src, dst=dst, ms=z(), mr=z(), R=z(),
                           o=np.zeros((cfgo.B, w.T, w.H, w.dv), np.float32))
    A, Bst = qs.new_state(cfgq), qs.new_state(cfgq)
    qs.qstate_init(cfgq, A, Bst)
    gst = qs.new_stats(cfgq)
    o = torch.zeros((w.B, w.T, w.H, w.dv), dtype=torch.float32, device="cuda")
    region, units, groups = cfgo.region_bytes, cfgo.units, cfgo.n_scale_groups
    report = []
    nwb = 0
    pool = ThreadPoolExecutor(max_workers=len(states)) if len(states) > 1 else None
    for wi, t0 in enumerate(range(0, w.T, w.C)):
        if max_wb is not None and wi >= max_wb:
            break
        t1 = min(w.T, t0 + w.C)
        gsrc, gdst = (A, Bst) if wi % 2 == 0 else (Bst, A)
        # inject the oracle's state (before this write-back) into the GPU
        for key, S in states.items():
            bsel = key if one else None
            kw = dict(b=key, region=region, units=units, groups=groups, H=w.H) if one else {}
            set_gpu_state(gsrc, S["src"], **kw)
            dst_meta = S["dst"].copy()
            set_gpu_state(gdst, dst_meta, **kw)
            for t, a in zip((gst.ema_s, gst.ema_r, gst.range), (S["ms"], S["mr"], S["R"])):
                if one:
                    t[key * units:(key + 1) * units].copy_(torch.from_numpy(a).cuda())
                else:
                    t.copy_(torch.from_numpy(a).cuda())
        qs.qstate_step(cfgq, gsrc, gdst, X, t0, t1, wi, o, gst)
        qs.qstate_check()
        g_out = from_gpu_state(orc, gdst)
        g_next = from_gpu_state(orc, gsrc)
        g_ms, g_mr, g_R = (host(t, np.float32) for t in (gst.ema_s, gst.ema_r, gst.range))
        og = host(o[:, t0:t1], np.float32)

        def orc_step(key):
            S = states[key]
            return orc.step(cfgo, S["src"], S["dst"], orc_inp[key], t0, t1, wi, S["o"], S["ms"], S["mr"],
                            S["R"], orc_code[key], s_lut, want_x=True, parallel=oracle_parallel)
        if len(states) > 1:
            xos = dict(zip(states, pool.map(orc_step, list(states))))
        else:
            xos = {key: orc_step(key) for key in states}
        for key, S in states.items():
            xo = xos[key]
            sl = (slice(key, key + 1) if one else slice(None))
            # readouts of this interval: normwise over the heads of each token, and per vector
            e_o = rel_err_tokens(og[sl], S["o"][:, t0:t1])
            e_v = rel_err_vectors(og[sl], S["o"][:, t0:t1])
            assert e_o <= REL_O_LOCKSTEP, (wi, key, e_o)
            assert e_v <= REL_O_QUANT, (wi, key, e_v)
            # packed state
            if one:
                gb = orc.Buf(g_out.payload[key * region:(key + 1) * region],
                             g_out.scales[key * groups:(key + 1) * groups],
                             g_out.widths[key * units:(key + 1) * units],
                             g_out.head_off[key * w.H:(key + 1) * w.H],
                             g_out.fidx[key * groups:(key + 1) * groups])
            else:
                gb = g_out
            us = slice(key * units, (key + 1) * units) if one else slice(None)
            st = compare_packed(orc, cfgo, gb, S["dst"], X=xo, R_gpu=g_R[us], R_ref=S["R"])
            # statistics
            for a, r in ((g_ms[us], S["ms"]), (g_mr[us], S["mr"])):
                assert np.allclose(a, r, rtol=REL_STATS, atol=1e-30), wi
            if cfgo.unit_kind == 0:
                assert np.allclose(g_R[us], S["R"], rtol=REL_STATS, atol=0), wi
            report.append(dict(wb=wi, b=key, rel_o=e_o, rel_o_vec=e_v, **st))
            # next widths: the oracle's allocation of its own statistics; the GPU's allocation
            # of the same statistics must agree bit for bit (checked through qstate_alloc_bits)
            wn, on = orc.alloc(cfgo, S["ms"], S["mr"], S["R"])
            sts = qs.Stats(dev(S["ms"], torch), dev(S["mr"], torch), dev(S["R"], torch))
            cq = qs.Config.from_workload(synth.scaled(w, B=cfgo.B), fit_every=fit_every,
                                         weight_kind=weight_kind)
            wt = torch.zeros(cfgo.B * units, dtype=torch.uint8, device="cuda")
            ot = torch.zeros(cfgo.B * w.H, dtype=torch.int32, device="cuda")
            qs.qstate_alloc_bits(cq, sts, wt, ot)
            assert np.array_equal(host(wt, np.uint8), wn) and np.array_equal(host(ot, np.uint32), on)
            # the GPU's own next widths (from its own statistics) agree almost everywhere
            agree = np.mean(g_next.widths[us] == wn)
            assert agree >= 0.99, (wi, key, agree)
            S["src"].widths[:], S["src"].head_off[:] = wn, on
            S["src"], S["dst"] = S["dst"], S["src"]
        nwb += 1
    if pool is not None:
        pool.shutdown()
    return report, {key: S["o"] for key, S in states.items()}


@pytest.mark.parametrize("name", ["tiny_kda", "kda_decode", "gdn_decode", "mamba2_decode", "kda_prefill"])
def test_quantised_lockstep(qs, orc, name):
    w = SMALL[name]
    rep, _ = _lockstep(qs, orc, w, log_decay=(w.gate_bits > 0))
    worst = max(r["rel_o"] for r in rep)
    worst_v = max(r["rel_o_vec"] for r in rep)
    agree = min(r["code_agree"] for r in rep)
    ties = sum(r["fidx_diff"] for r in rep)
    print(f"{name}: {len(rep)} write-backs, worst rel readout {worst:.2e} per token "
          f"({worst_v:.2e} per vector), min code agreement {agree:.6f}, near-tie factor "
          f"differences {ties}")


def test_quantised_lockstep_fit_every(qs, orc):
    w = small("kda_decode", B=2, H=4, T=10, gate_bits=0)
    _lockstep(qs, orc, w, fit_every=4)


@pytest.mark.parametrize("dk,dv", [(128, 128)] + HEAD_SHAPES)
@pytest.mark.parametrize("fit_every", [1, 3])
def test_quantised_lockstep_head_unit_shapes(qs, orc, dk, dv, fit_every):
    """Gated DeltaNet (head unit) write-backs at every state shape, refitting every write-back
    or reusing the stored factors between refits."""
    w = small("gdn_decode", B=2, H=4, T=8, dk=dk, dv=dv)
    _lockstep(qs, orc, w, fit_every=fit_every)


def test_persistent_decay_lockstep(qs, orc):
    """KDA with per-channel decay fixed over tokens (slow channels, log-quantised rates)."""
    w = synth.scaled(synth.EXTENSION_WORKLOADS["kda_persistent"], B=3, H=4, T=12)
    _lockstep(qs, orc, w, log_decay=True)


@pytest.mark.parametrize("name,log_decay,form", [("kda_decode", True, 0), ("mamba2_decode", False, 0),
                                                 ("kda_prefill", False, 0), ("kda_prefill", False, 1)])
def test_current_allocation_lockstep(qs, orc, name, log_decay, form):
    """alloc_mode current: each write-back allocates from its own statistics (a statistics
    pass, the allocation, then the packing pass).  The oracle runs free; before every
    write-back its state is copied into the GPU; widths, codes, readouts and statistics of the
    GPU's write-back are compared with the oracle's.  form 1: both passes in chunked form."""
    w = SMALL[name]
    cfgq = qs.Config.from_workload(w, alloc_mode=1, interval_form=form)
    cfgo = orc.Cfg.from_workload(w, alloc_mode=1)
    inp = synth.host_inputs(w)
    s_code = s_lut = None
    if log_decay:
        nchan = w.H * w.dk if w.per_row_decay else w.H
        s_code, s_lut, _ = orc.quant_decay(inp["s"], nchan, w.gate_bits)
    X, _ = _dev_inputs(w, inp, qs, s_code, s_lut)
    src, dst = orc.init_state(cfgo)
    z = lambda: np.zeros(cfgo.B * cfgo.units, np.float32)
    ms, mr, R = z(), z(), z()
    oo = np.zeros((w.B, w.T, w.H, w.dv), np.float32)
    A, Bst = qs.new_state(cfgq), qs.new_state(cfgq)
    qs.qstate_init(cfgq, A, Bst)
    gst = qs.new_stats(cfgq)
    o = torch.zeros((w.B, w.T, w.H, w.dv), dtype=torch.float32, device="cuda")
    for wi, t0 in enumerate(range(0, w.T, w.C)):
        t1 = min(w.T, t0 + w.C)
        gsrc, gdst = (A, Bst) if wi % 2 == 0 else (Bst, A)
        set_gpu_state(gsrc, src)
        for t, a in zip((gst.ema_s, gst.ema_r, gst.range), (ms, mr, R)):
            t.copy_(torch.from_numpy(a).cuda())
        qs.qstate_step(cfgq, gsrc, gdst, X, t0, t1, wi, o, gst)
        qs.qstate_check()
        xo = orc.step(cfgo, src, dst, inp, t0, t1, wi, oo, ms, mr, R, s_code, s_lut, want_x=True)
        g_out = from_gpu_state(orc, gdst)
        assert np.array_equal(g_out.widths, dst.widths), wi      # allocated from this write-back
        assert np.array_equal(g_out.head_off, dst.head_off), wi
        compare_packed(orc, cfgo, g_out, dst, X=xo)
        og = host(o[:, t0:t1], np.float32)
        assert rel_err_tokens(og, oo[:, t0:t1]) <= REL_O_LOCKSTEP
        assert rel_err_vectors(og, oo[:, t0:t1]) <= REL_O_QUANT
        for g, r in ((gst.ema_s, ms), (gst.ema_r, mr), (gst.range, R)):
            assert np.allclose(host(g, np.float32), r, rtol=REL_STATS, atol=1e-30), wi
        src, dst = dst, src


@pytest.mark.parametrize("name", ["kda_general", "gdn_general"])
def test_general_erasure_lockstep(qs, orc, name):
    """Eq. (1) with a and w given per token (row unit and head unit) stays in lockstep."""
    w = synth.scaled(synth.EXTENSION_WORKLOADS[name], B=3, H=4, T=10)
    _lockstep(qs, orc, w)


@pytest.mark.parametrize("name", ["kda_general", "gdn_general"])
def test_general_erasure_fp32_free_running(qs, orc, name):
    """The unquantised FP32 recurrence with general a and w against the oracle's recurrence."""
    w = synth.scaled(synth.EXTENSION_WORKLOADS[name], B=2, H=3, T=64)
    cfgq, cfgo = qs.Config.from_workload(w), orc.Cfg.from_workload(w)
    inp = synth.host_inputs(w)
    X, _ = _dev_inputs(w, inp, qs)
    S = torch.zeros((w.B, w.H, w.dk, w.dv), dtype=torch.float32, device="cuda")
    o = torch.zeros((w.B, w.T, w.H, w.dv), dtype=torch.float32, device="cuda")
    qs.qstate_scan_fp32(cfgq, S, X, 0, w.T, o)
    qs.qstate_check()
    og = host(o, np.float32)
    worst = 0.0
    for b in range(w.B):
        for h in range(w.H):
            o32, _ = orc.recur(np.zeros((w.dk, w.dv)), *orc.expand_inputs(cfgo, inp, b, h), dtype=np.float32)
            worst = max(worst, rel_err_vectors(og[b, :, h], o32))
    assert worst <= REL_O_FP32


@pytest.mark.parametrize("kind", [5, 7])
def test_quantised_lockstep_weight_kinds(qs, orc, kind):
    """A scan with the write-back-factor or shuffled-decay weights (Table 1) stays in lockstep:
    the allocation between write-backs uses the configured weight."""
    _lockstep(qs, orc, SMALL["kda_decode"], log_decay=True, weight_kind=kind)


CHUNKED_ROW_CASES = {
    "coded_g2": (lambda: small("kda_decode", B=2, H=3, T=19, C=8), True),
    "coded_g3": (lambda: small("kda_decode", B=2, H=3, T=13, C=5, gate_bits=3), True),
    "mamba2": (lambda: small("mamba2_decode", B=2, H=16, T=17, C=8), False),
    "tiny": (lambda: small("tiny_kda", T=23, C=7), False),
    "general": (lambda: synth.scaled(synth.EXTENSION_WORKLOADS["kda_general"], B=2, H=3, T=20, C=6), False),
    "persistent": (lambda: synth.scaled(synth.EXTENSION_WORKLOADS["kda_persistent"], B=2, H=3, T=14, C=4), True),
}


@pytest.mark.parametrize("case", sorted(CHUNKED_ROW_CASES))
def test_quantised_lockstep_chunked_row_kernel(qs, orc, case):
    """Write-back periods C > 1 through the row-unit kernel, whose tokens after the first take
    their inputs from alternating buffers filled one token ahead: log-coded rates from the
    head's level table (g = 2) and from the global table (g = 3), per-head rates without
    erasure (Mamba-2, dv = 64), 64 x 64 heads, general a and w, persistent decay; every case
    ends on a ragged interval."""
    make, log_decay = CHUNKED_ROW_CASES[case]
    w = make()
    assert w.C > 1 and w.T % w.C != 0
    _lockstep(qs, orc, w, log_decay=log_decay)


@pytest.mark.parametrize("name,kw", [("kda_decode", dict(B=2, H=3, T=6)),
                                     ("gdn_decode", dict(B=2, H=4, T=6)),
                                     ("kda_prefill", dict(B=1, H=2, T=40, C=16))])
def test_quantised_lockstep_wide_rows(qs, orc, name, kw):
    """The widest rows (14 bits on average, widths up to 16) token by token, row unit (KDA)
    and head unit (Gated DeltaNet); codes of rows wider than 8 bits are checked per code."""
    w = small(name, bbar=14, bmin=0, bmax=16, gate_bits=0, **kw)
    _lockstep(qs, orc, w)


def test_quantised_lockstep_ragged_chunks(qs, orc):
    w = small("kda_prefill", B=1, H=2, T=37, C=16)
    _lockstep(qs, orc, w)


@pytest.mark.parametrize("name,T,sample", [("kda_decode", 3, (0, 131, 255)),
                                           ("gdn_decode", 3, (0, 63)),
                                           ("mamba2_decode", 2, (5, 127)),
                                           ("kda_prefill", 70, (0, 15))])
def test_full_size_sampled_lockstep(qs, orc, name, T, sample):
    """Full batch and heads of the benchmark workloads, in the launch configuration the
    benchmark times; sampled batch elements are compared write-back by write-back."""
    w = synth.scaled(synth.WORKLOADS[name], T=T)
    _lockstep(qs, orc, w, log_decay=(w.gate_bits > 0), sample_b=sample)


def test_tiny_kda_full_lockstep(qs, orc):
    """The tiny recurrence at its full length (T = 256 per-token write-backs)."""
    _lockstep(qs, orc, synth.WORKLOADS["tiny_kda"])


# ---------------------------------------------------------------------------------- edge cases
def test_inconsistent_layout_is_reported(qs, orc):
    w = small("kda_decode", B=2, H=2, T=2, gate_bits=0)
    cfgq = qs.Config.from_workload(w)
    inp = synth.host_inputs(w)
    X, _ = _dev_inputs(w, inp, qs)
    A, Bst = qs.new_state(cfgq), qs.new_state(cfgq)
    qs.qstate_init(cfgq, A, Bst)
    Bst.widths[5] = 17                      # caught by the kernel's own layout check
    o = torch.zeros((w.B, w.T, w.H, w.dv), dtype=torch.float32, device="cuda")
    qs.qstate_step(cfgq, A, Bst, X, 0, 1, 0, o, qs.new_stats(cfgq))
    with pytest.raises(qs.QstateError) as e:
        qs.qstate_check()
    assert e.value.code == qs.QSTATE_EDEVICE
    qs.qstate_check()                       # cleared


def test_host_side_argument_errors(qs):
    cfg = qs.Config.from_workload(small("kda_decode", B=1, H=2, T=2))
    A, Bst = qs.new_state(cfg), qs.new_state(cfg)
    o = torch.zeros((1, 2, 2, 128), device="cuda")
    z = torch.zeros((1, 2, 2, 128), device="cuda")
    X = qs.Inputs(z, z, z, None, None, None, torch.zeros((1, 2, 2), device="cuda"), 2)
    with pytest.raises(qs.QstateError):
        qs.qstate_step(cfg, A, Bst, X, 0, 1, 0, o, qs.new_stats(cfg))   # no decay rates
    X.s = torch.ones((1, 2, 2, 128), device="cuda")
    with pytest.raises(qs.QstateError):
        qs.qstate_step(cfg, A, Bst, X, 0, 2, 0, o, qs.new_stats(cfg))   # 2 tokens > C = 1
    bad = qs.Config.from_workload(small("kda_decode", B=1, H=2, T=2), bmin=5)
    with pytest.raises(qs.QstateError) as e:
        qs.qstate_init(bad, A, Bst)
    assert e.value.code == qs.QSTATE_EBUDGET


def test_scan_equals_repeated_steps(qs, orc):
    """qstate_scan = the sequence of qstate_step calls, bit for bit."""
    w = small("kda_prefill", B=2, H=2, T=40, C=16)
    cfgq = qs.Config.from_workload(w)
    inp = synth.host_inputs(w)
    X, _ = _dev_inputs(w, inp, qs)
    outs = []
    for mode in ("scan", "steps"):
        A, Bst = qs.new_state(cfgq), qs.new_state(cfgq)
        qs.qstate_init(cfgq, A, Bst)
        st = qs.new_stats(cfgq)
        o = torch.zeros((w.B, w.T, w.H, w.dv), dtype=torch.float32, device="cuda")
        if mode == "scan":
            pong = qs.qstate_scan(cfgq, A, Bst, X, 0, w.T, 0, o, st)
            fin = Bst if pong else A
        else:
            src, dst = A, Bst
            for wi, t0 in enumerate(range(0, w.T, w.C)):
                qs.qstate_step(cfgq, src, dst, X, t0, min(w.T, t0 + w.C), wi, o, st)
                src, dst = dst, src
            fin = src
        qs.qstate_check()
        outs.append((host(o, np.float32), from_gpu_state(orc, fin)))
    assert np.array_equal(outs[0][0], outs[1][0])
    for f in ("payload", "scales", "widths", "head_off", "fidx"):
        assert np.array_equal(getattr(outs[0][1], f), getattr(outs[1][1], f))


# ------------------------------------------------------------------ host-staged scan
@pytest.mark.parametrize("name,chunk,form", [("kda_decode", 3, 0), ("gdn_decode", 4, 0), ("kda_prefill", 8, 0),
                                             ("kda_prefill", 8, 1)])
def test_scan_host_equals_scan(qs, orc, name, chunk, form):
    """qstate_scan_host (inputs copied from pinned host memory chunk by chunk on a second
    stream) gives qstate_scan's readouts and final state bit for bit (form 1: both in chunked
    form)."""
    w = SMALL[name]
    if name == "kda_prefill":
        w = synth.scaled(w, T=2 * w.C + 5)
        chunk = w.C
    cfgq = qs.Config.from_workload(w, interval_form=form)
    inp = synth.host_inputs(w)
    s_code = s_lut = None
    if w.gate_bits:
        nchan = w.H * w.dk if w.per_row_decay else w.H
        s_code, s_lut, _ = orc.quant_decay(inp["s"], nchan, w.gate_bits)
    X, _ = _dev_inputs(w, inp, qs, s_code, s_lut)
    # reference: device inputs
    A, Bs, st = qs.new_state(cfgq), qs.new_state(cfgq), qs.new_stats(cfgq)
    qs.qstate_init(cfgq, A, Bs)
    o_ref = torch.zeros((w.B, w.T, w.H, w.dv), dtype=torch.float32, device="cuda")
    pong_ref = qs.qstate_scan(cfgq, A, Bs, X, 0, w.T, 0, o_ref, st)
    qs.qstate_check()
    # host-staged: device buffers start as garbage and are filled chunk by chunk
    pin = lambda a: torch.from_numpy(np.ascontiguousarray(a)).pin_memory()
    xh = qs.Inputs(pin(inp["q"]), pin(inp["k"]), pin(inp["v"]),
                   None if s_code is not None else pin(inp["s"]), None, None,
                   pin(inp["beta"]) if w.erase else None, w.T)
    xd = qs.Inputs(torch.full_like(X.q, 7.0), torch.full_like(X.k, 7.0), torch.full_like(X.v, 7.0),
                   None if X.s is None else torch.full_like(X.s, 7.0), X.s_code, X.s_lut,
                   None if X.beta is None else torch.full_like(X.beta, 7.0), w.T)
    A2, B2, st2 = qs.new_state(cfgq), qs.new_state(cfgq), qs.new_stats(cfgq)
    qs.qstate_init(cfgq, A2, B2)
    o_dev = torch.zeros_like(o_ref)
    o_host = torch.zeros(o_ref.shape, dtype=torch.float32).pin_memory()
    s1, s2 = torch.cuda.Stream(), torch.cuda.Stream()
    s1.wait_stream(torch.cuda.current_stream())
    pong = qs.qstate_scan_host(cfgq, A2, B2, xh, xd, 0, w.T, 0, o_host, o_dev, st2, chunk, s1, s2)
    s1.synchronize()
    qs.qstate_check()
    assert pong == pong_ref
    assert np.array_equal(o_host.numpy().view(np.uint32), host(o_ref, np.float32).view(np.uint32))
    fin, fin2 = (Bs, B2) if pong else (A, A2)
    for f in ("payload", "scales", "widths", "head_off", "fidx"):
        assert torch.equal(getattr(fin, f), getattr(fin2, f)), f
    for f in ("ema_s", "ema_r", "range"):
        assert torch.equal(getattr(st, f), getattr(st2, f)), f


def test_scan_host_argument_errors(qs):
    w = SMALL["kda_decode"]
    cfgq = qs.Config.from_workload(w, gate_bits=0)
    inp = synth.host_inputs(w)
    X, _ = _dev_inputs(w, inp, qs)
    A, Bs, st = qs.new_state(cfgq), qs.new_state(cfgq), qs.new_stats(cfgq)
    xh = qs.Inputs(*(torch.from_numpy(np.ascontiguousarray(inp[n])) for n in ("q", "k", "v", "s")),
                   None, None, torch.from_numpy(np.ascontiguousarray(inp["beta"])), w.T)
    o = torch.zeros((w.B, w.T, w.H, w.dv), dtype=torch.float32, device="cuda")
    oh = torch.zeros(o.shape, dtype=torch.float32)
    s1 = torch.cuda.Stream()
    with pytest.raises(qs.QstateError):        # one stream for both roles
        qs.qstate_scan_host(cfgq, A, Bs, xh, X, 0, w.T, 0, oh, o, st, 2, s1, s1)
    with pytest.raises(qs.QstateError):        # chunk not a multiple of C (C = 1: chunk 0)
        qs.qstate_scan_host(cfgq, A, Bs, xh, X, 0, w.T, 0, oh, o, st, 0, s1, torch.cuda.Stream())


@pytest.mark.parametrize("form", [0, 1])
def test_empty_token_range(qs, form):
    """An empty token range [t, t) is a no-op for qstate_scan and qstate_scan_host (state,
    statistics and readouts untouched, the state stays in ping) and an error for qstate_step,
    whose interval holds 1..C tokens; reversed or out-of-range ranges are errors."""
    w = small("kda_prefill", B=2, H=2, T=40, C=16)
    cfgq = qs.Config.from_workload(w, interval_form=form)
    inp = synth.host_inputs(w)
    X, _ = _dev_inputs(w, inp, qs)
    A, Bs, st = qs.new_state(cfgq), qs.new_state(cfgq), qs.new_stats(cfgq)
    qs.qstate_init(cfgq, A, Bs)
    qs.qstate_scan(cfgq, A, Bs, X, 0, w.C, 0, torch.zeros((w.B, w.T, w.H, w.dv), device="cuda"), st)
    torch.cuda.synchronize()
    fields = ("payload", "scales", "widths", "head_off", "fidx")
    snap = {(n, f): getattr(s, f).clone() for n, s in (("A", A), ("B", Bs)) for f in fields}
    snap_st = {f: getattr(st, f).clone() for f in ("ema_s", "ema_r", "range")}
    o = torch.full((w.B, w.T, w.H, w.dv), 3.0, device="cuda")
    assert not qs.qstate_scan(cfgq, A, Bs, X, 7, 7, 1, o, st)
    oh = torch.full(o.shape, 3.0).pin_memory()
    s1, s2 = torch.cuda.Stream(), torch.cuda.Stream()
    s1.wait_stream(torch.cuda.current_stream())
    xh = qs.Inputs(*(torch.from_numpy(np.ascontiguousarray(inp[n])).pin_memory() for n in ("q", "k", "v", "s")),
                   None, None, torch.from_numpy(np.ascontiguousarray(inp["beta"])).pin_memory(), w.T)
    assert not qs.qstate_scan_host(cfgq, A, Bs, xh, X, 7, 7, 1, oh, o, st, w.C, s1, s2)
    s1.synchronize()
    qs.qstate_check()
    for (n, f), v in snap.items():
        assert torch.equal(getattr(A if n == "A" else Bs, f), v), (n, f)
    for f, v in snap_st.items():
        assert torch.equal(getattr(st, f), v), f
    assert bool((o == 3.0).all()) and bool((oh == 3.0).all())
    for t0, t1 in ((7, 7), (9, 8)):
        with pytest.raises(qs.QstateError) as e:
            qs.qstate_step(cfgq, A, Bs, X, t0, t1, 1, o, st)
        assert e.value.code == qs.QSTATE_EINVAL
    for t0, t1 in ((9, 8), (0, w.T + 1), (-1, 3)):
        with pytest.raises(qs.QstateError) as e:
            qs.qstate_scan(cfgq, A, Bs, X, t0, t1, 1, o, st)
        assert e.value.code == qs.QSTATE_EINVAL
