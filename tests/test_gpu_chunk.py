"""The chunked form of a write-back interval (tensor cores, 16-token blocks) against the
oracle's token-by-token recurrence: quantised write-backs in lockstep (codes >= 99.99 %
identical and within one step, readouts and statistics within 1e-5), intervals that
are whole blocks, ragged blocks and single tokens, log-coded and per-head rates, no erasure,
the full prefill batch, and the status raised when a block's decay leaves the form's range."""
import numpy as np
import pytest

import synth
from parity import from_gpu_state, host
from test_gpu_parity import _dev_inputs, _lockstep, small

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")

CHUNK = 1

CASES = {
    # interval = 4 whole blocks, then a ragged 22-token interval (a block of 16 and one of 6)
    "prefill_c64": (lambda: small("kda_prefill", B=2, H=3, T=150, C=64), False),
    # intervals of 40 tokens: two blocks and a half block
    "prefill_c40": (lambda: small("kda_prefill", B=2, H=3, T=100, C=40), False),
    # one block per interval, and intervals shorter than a block
    "prefill_c16": (lambda: small("kda_prefill", B=1, H=4, T=48, C=16), False),
    "prefill_c5": (lambda: small("kda_prefill", B=1, H=3, T=17, C=5), False),
    # log-quantised rates from the head's level table
    "decode_coded_c32": (lambda: small("kda_decode", B=2, H=3, T=70, C=32), True),
    # per-head rates, delta rule, row unit at 128 x 128
    "gdn_row_c24": (lambda: synth.scaled(synth.WORKLOADS["gdn_decode"], B=2, H=4, T=50, C=24,
                                         unit="row", bmin=1, bmax=8), False),
    # no erasure (a = 0, w = 1), per-head rates, 128 x 128
    "mamba_128_c32": (lambda: synth.scaled(synth.WORKLOADS["mamba2_decode"], B=2, H=8, T=70, C=32,
                                           dv=128, group_heads=4), False),
    # log-quantised rates with 8 levels (level table read from global memory)
    "decode_coded_g3_c48": (lambda: small("kda_decode", B=2, H=3, T=70, C=48, gate_bits=3), True),
    # per-head log-quantised rates, row unit
    "gdn_row_coded_c32": (lambda: synth.scaled(synth.WORKLOADS["gdn_decode"], B=2, H=4, T=45, C=32,
                                               unit="row", bmin=1, bmax=8, gate_bits=2), True),
    # the widest rows (14 bits on average, widths 12..16 allocated): the largest payload
    # buffer the chunked form's shared memory holds
    "prefill_wide_c32": (lambda: small("kda_prefill", B=2, H=3, T=70, C=32, bbar=14, bmin=0, bmax=16), False),
    # slow channels that keep their rate over the whole sequence
    "persistent_c64": (lambda: synth.scaled(synth.EXTENSION_WORKLOADS["kda_persistent"], B=2, H=3,
                                            T=130, C=64), True),
}


@pytest.mark.parametrize("case", sorted(CASES))
def test_chunked_form_lockstep(qs, orc, case):
    make, log_decay = CASES[case]
    w = make()
    rep, _ = _lockstep(qs, orc, w, log_decay=log_decay, interval_form=CHUNK)
    worst = max(r["rel_o"] for r in rep)
    worst_v = max(r["rel_o_vec"] for r in rep)
    agree = min(r["code_agree"] for r in rep)
    wide = min((r["wide_code_agree"] for r in rep if "wide_code_agree" in r), default=None)
    print(f"{case}: {len(rep)} write-backs, worst rel readout {worst:.2e} per token ({worst_v:.2e} "
          f"per vector), min code agreement {agree:.6f}"
          + ("" if wide is None else f", rows wider than 8 bits {wide:.6f}"))


def test_chunked_form_refit_schedule(qs, orc):
    w = small("kda_prefill", B=2, H=4, T=96, C=32)
    _lockstep(qs, orc, w, fit_every=3, interval_form=CHUNK)


def test_chunked_form_full_prefill_batch_sampled(qs, orc):
    """All 16 x 32 heads of the prefill workload in the launch configuration the benchmark
    times (one CTA per SM, persistent); two sampled batch elements compared write-back by
    write-back, the second interval ragged."""
    w = synth.scaled(synth.WORKLOADS["kda_prefill"], T=70)
    _lockstep(qs, orc, w, sample_b=(0, 15), interval_form=CHUNK)


def test_chunked_form_scan_equals_steps(qs, orc):
    """qstate_scan in chunked form = its sequence of qstate_step calls, bit for bit."""
    w = small("kda_prefill", B=2, H=2, T=72, C=32)
    cfgq = qs.Config.from_workload(w, interval_form=CHUNK)
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


def test_chunked_form_decay_out_of_range_is_reported(qs, orc):
    """Rates summing past the FP32 range over a 16-token block (here 10 per token) are
    reported through the device status; the token form takes the same inputs."""
    w = small("kda_prefill", B=1, H=2, T=32, C=32)
    inp = synth.host_inputs(w)
    inp["s"] = np.full_like(inp["s"], 10.0)
    for form, bad in ((0, False), (CHUNK, True)):
        cfgq = qs.Config.from_workload(w, interval_form=form)
        X, _ = _dev_inputs(w, inp, qs)
        A, Bst = qs.new_state(cfgq), qs.new_state(cfgq)
        qs.qstate_init(cfgq, A, Bst)
        st = qs.new_stats(cfgq)
        o = torch.zeros((w.B, w.T, w.H, w.dv), dtype=torch.float32, device="cuda")
        qs.qstate_step(cfgq, A, Bst, X, 0, w.T, 0, o, st)
        if bad:
            with pytest.raises(qs.QstateError) as e:
                qs.qstate_check()
            assert e.value.code == qs.QSTATE_EDEVICE
            assert b"16-token block" in qs.load().qstate_last_error()
        else:
            qs.qstate_check()



def test_chunked_form_timeout_is_reported(qs, orc):
    """The chunked form's bounded waits for its tensor-core products: with a wait limit of 0
    polls every wait gives up at once while the products still complete, the status reports
    QSTATE_ETIMEOUT (not a generic device error), and the next call with the default limit
    gives the clean run's results bit for bit (tensor memory was freed only once the products
    had finished)."""
    w = small("kda_prefill", B=2, H=3, T=40, C=40)
    cfgq = qs.Config.from_workload(w, interval_form=CHUNK)
    inp = synth.host_inputs(w)
    X, _ = _dev_inputs(w, inp, qs)

    def run():
        A, Bst = qs.new_state(cfgq), qs.new_state(cfgq)
        qs.qstate_init(cfgq, A, Bst)
        st = qs.new_stats(cfgq)
        o = torch.zeros((w.B, w.T, w.H, w.dv), dtype=torch.float32, device="cuda")
        qs.qstate_step(cfgq, A, Bst, X, 0, w.T, 0, o, st)
        return o, Bst, A, st

    clean = run()
    qs.qstate_check()
    qs.qstate_set_wait_limit(0)
    try:
        run()
        with pytest.raises(qs.QstateError) as e:
            qs.qstate_check()
        assert e.value.code == qs.QSTATE_ETIMEOUT
        assert b"timed out" in qs.load().qstate_last_error()
    finally:
        qs.qstate_set_wait_limit(-1)
    again = run()
    qs.qstate_check()
    assert torch.equal(clean[0], again[0])
    for i in (1, 2):
        for f in ("payload", "scales", "widths", "head_off", "fidx"):
            assert torch.equal(getattr(clean[i], f), getattr(again[i], f)), f
    for f in ("ema_s", "ema_r", "range"):
        assert torch.equal(getattr(clean[3], f), getattr(again[3], f)), f
