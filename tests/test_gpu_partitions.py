"""A scan run as concurrent batch partitions (qstate_set_scan_partitions) gives the results of
one chain bit for bit (GPU).

The batch elements are independent problems (Eq. 1 and the allocation of Sec. 3 act on each
element's own state and budget), and every kernel computes each head and batch element on its
own, so splitting the batch over streams may change the timing only.  Uneven splits (B = 5 over
2, 3 and 4 partitions) and more partitions than batch elements are covered, for the token form,
the chunked form, the head unit, the 128 x 64 and 64 x 64 shapes, general erasure and the
current-range allocation.
"""
import numpy as np
import pytest

import synth
from test_gpu_parity import _dev_inputs

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")

# id -> (workload, log-coded rates, interval form, extra configuration); T and H chosen so that
# every per-element array offset is a multiple of 16 bytes (the partitions then start where asked)
def _w(name, **kw):
    base = synth.WORKLOADS.get(name) or synth.EXTENSION_WORKLOADS[name]
    return synth.scaled(base, B=5, **kw)


CASES = {
    "kda_decode": (lambda: _w("kda_decode", H=8, T=48), True, 0, {}),
    "kda_prefill": (lambda: _w("kda_prefill", H=8, T=80), False, 1, {}),
    "gdn_decode": (lambda: _w("gdn_decode", H=16, T=48), False, 0, {}),
    "mamba2_decode": (lambda: _w("mamba2_decode", H=8, T=32), False, 0, {}),
    "kda_64x64": (lambda: _w("tiny_kda", H=4, T=40), False, 0, {}),
    "kda_general": (lambda: _w("kda_general", H=4, T=24), False, 0, {}),
    "gdn_general": (lambda: _w("gdn_general", H=16, T=24), False, 0, {}),
    "kda_alloc_current": (lambda: _w("kda_decode", H=8, T=24), True, 0, {"alloc_mode": 1}),
}


def _scan(qs, orc, w, log_decay, form, parts, stream=None, extra=None):
    qs.qstate_set_scan_partitions(parts)
    try:
        inp = synth.host_inputs(w)
        s_code = s_lut = None
        if log_decay:
            nchan = w.H * w.dk if w.per_row_decay else w.H
            s_code, s_lut, _ = orc.quant_decay(inp["s"], nchan, w.gate_bits)
        cfg = qs.Config.from_workload(w, interval_form=form, **(extra or {}))
        X, _ = _dev_inputs(w, inp, qs, s_code, s_lut)
        A, Bs = qs.new_state(cfg), qs.new_state(cfg)
        qs.qstate_init(cfg, A, Bs)
        st = qs.new_stats(cfg)
        o = torch.zeros((w.B, w.T, w.H, w.dv), dtype=torch.float32, device="cuda")
        used = qs.qstate_scan_partition_count(cfg, X, st)
        if stream is None:
            flip = qs.qstate_scan(cfg, A, Bs, X, 0, w.T, 0, o, st)
            qs.qstate_check()
        else:
            with torch.cuda.stream(stream):
                flip = qs.qstate_scan(cfg, A, Bs, X, 0, w.T, 0, o, st, stream)
            # the join orders every partition before the caller's stream continues
            done = torch.empty(1, device="cuda")
            with torch.cuda.stream(stream):
                done.copy_(o.abs().sum().reshape(1))
            qs.qstate_check(stream)
            torch.cuda.synchronize()
            assert np.isfinite(done.cpu().numpy()).all()
    finally:
        qs.qstate_set_scan_partitions(0)
    bufs = {}
    for tag, S in (("A", A), ("B", Bs)):
        for f in ("payload", "scales", "widths", "head_off", "fidx"):
            bufs[f"{tag}.{f}"] = getattr(S, f).cpu().numpy().copy()
    for f in ("ema_s", "ema_r", "range"):
        t = getattr(st, f)
        if t is not None:
            bufs[f] = t.cpu().numpy().view(np.uint32).copy()
    bufs["o"] = o.cpu().numpy().view(np.uint32).copy()
    return flip, bufs, used


@pytest.mark.parametrize("name", list(CASES))
def test_partitioned_scan_is_bit_identical(qs, orc, name):
    make, log_decay, form, extra = CASES[name]
    w = make()
    flip1, ref, used1 = _scan(qs, orc, w, log_decay, form, 1, extra=extra)
    assert used1 == 1
    for parts in (2, 3, 4, 8):
        flip, got, used = _scan(qs, orc, w, log_decay, form, parts, extra=extra)
        assert used == min(parts, w.B)     # every partition start is 16-byte aligned here
        assert flip == flip1
        for key in ref:
            assert np.array_equal(got[key], ref[key]), (parts, key)


def test_partitioned_scan_on_a_caller_stream(qs, orc):
    # the caller's own (non-default) stream: the work after the call is ordered after every
    # partition's
    w = synth.scaled(synth.WORKLOADS["kda_prefill"], B=4, H=8, T=80)
    _, ref, _ = _scan(qs, orc, w, False, 1, 1)
    s = torch.cuda.Stream()
    _, got, used = _scan(qs, orc, w, False, 1, 4, stream=s)
    assert used == 4
    for key in ref:
        assert np.array_equal(got[key], ref[key]), key

