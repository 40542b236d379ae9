"""Readout error of the quantised recurrence under the paper's allocation (GPU, end to end).

A synthetic KDA recurrence whose key channels keep their decay rate over the whole sequence,
log-uniform in [1e-3, 1] (some channels remember for a thousand tokens, some for one), is run
through the library at a two-bit mean payload with chunked write-back (C = 64 and 16), the
setting of the synthetic readout experiment of Sec. 1 (Fig. 1(d)) and of the chunked ablation
of Table 1, and at a four-bit mean with per-token write-back (C = 1, Table 2a).
The readouts are compared with the library's unquantised FP32 recurrence on the same inputs:

    relative readout MSE = sum (o - o_fp32)^2 / sum o_fp32^2.

Widths from the allocation of Eq. 3-4 must give a much smaller error than uniform widths (the
claim of Sec. 3 and Table 1), and the GPU's free-running error must agree with the oracle's
own free-running scan of the same configuration (which the parity tests pin step by step).
"""
import numpy as np
import pytest

import synth

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")


def _workload(C, bbar, bmin, bmax, T):
    return synth.Workload(f"kda_persistent_c{C}", synth.KDA, B=2, H=2, dk=128, dv=128, T=T, C=C,
                          bbar=bbar, bmin=bmin, bmax=bmax, unit="row", gate_bits=0,
                          persistent=1e-3, seed=9000)


def _gpu_rel_mse(qs, w, weight_kind, o_ref, form=0):
    cfg = qs.Config.from_workload(w, weight_kind=weight_kind, interval_form=form)
    inp = synth.host_inputs(w)
    d = {k: torch.from_numpy(v).cuda() for k, v in inp.items()}
    X = qs.Inputs(d["q"], d["k"], d["v"], d["s"], None, None, d["beta"], w.T)
    A, Bst = qs.new_state(cfg), qs.new_state(cfg)
    qs.qstate_init(cfg, A, Bst)
    st = qs.new_stats(cfg)
    o = torch.zeros((w.B, w.T, w.H, w.dv), dtype=torch.float32, device="cuda")
    qs.qstate_scan(cfg, A, Bst, X, 0, w.T, 0, o, st)
    qs.qstate_check()
    og = o.cpu().numpy().astype(np.float64)
    return float(np.sum((og - o_ref) ** 2) / np.sum(o_ref ** 2))


def _gpu_fp32_readouts(qs, w):
    cfg = qs.Config.from_workload(w)
    inp = synth.host_inputs(w)
    d = {k: torch.from_numpy(v).cuda() for k, v in inp.items()}
    X = qs.Inputs(d["q"], d["k"], d["v"], d["s"], None, None, d["beta"], w.T)
    S = torch.zeros((w.B, w.H, w.dk, w.dv), dtype=torch.float32, device="cuda")
    o = torch.zeros((w.B, w.T, w.H, w.dv), dtype=torch.float32, device="cuda")
    qs.qstate_scan_fp32(cfg, S, X, 0, w.T, o)
    qs.qstate_check()
    return o.cpu().numpy().astype(np.float64)


# (C, bbar, bmin, bmax, T, bound on ours / uniform): chunked write-back at a two-bit mean payload
# (Fig. 1(d), Table 1) and per-token write-back at a four-bit mean (Table 2a); the oracle gives
# 0.30, 0.31 and 0.21 for the error ratio on these inputs
CASES = [(64, 2, 1, 8, 512, 0.5, 0), (16, 2, 1, 8, 512, 0.5, 0), (1, 4, 0, 8, 256, 0.4, 0),
         # the chunked form of the write-back intervals (tensor cores)
         (64, 2, 1, 8, 512, 0.5, 1), (16, 2, 1, 8, 512, 0.5, 1)]


@pytest.mark.parametrize("C,bbar,bmin,bmax,T,ratio,form", CASES)
def test_allocation_lowers_readout_error(qs, orc, C, bbar, bmin, bmax, T, ratio, form):
    W = _workload(C, bbar, bmin, bmax, T)
    o_ref = _gpu_fp32_readouts(qs, W)
    errs = {name: _gpu_rel_mse(qs, W, kind, o_ref, form)
            for name, kind in (("uniform", qs.WEIGHT_UNIFORM), ("ours", qs.WEIGHT_OURS),
                               ("range", qs.WEIGHT_RANGE), ("persistence", qs.WEIGHT_PERSIST))}
    print("relative readout MSE:", ", ".join(f"{k} {v:.4e}" for k, v in errs.items()))
    assert errs["ours"] < ratio * errs["uniform"], errs
    assert errs["ours"] < errs["range"], errs
    # the oracle's own free-running scan of the same configuration gives the same error
    o_orc, *_ = orc.scan(orc.Cfg.from_workload(W), synth.host_inputs(W))
    e_orc = float(np.sum((o_orc.astype(np.float64) - o_ref) ** 2) / np.sum(o_ref ** 2))
    print(f"oracle, Eq. 3 widths: {e_orc:.4e}")
    assert abs(errs["ours"] - e_orc) <= 0.05 * e_orc, (errs["ours"], e_orc)


def _fp32_readouts_with_rates(qs, w, inp, s_code=None, s_lut=None, g=0):
    """The library's unquantised recurrence, with exact rates or with coded rates + levels."""
    cfg = qs.Config.from_workload(w, gate_bits=g)
    d = {k: torch.from_numpy(v).cuda() for k, v in inp.items()}
    if s_code is None:
        X = qs.Inputs(d["q"], d["k"], d["v"], d["s"], None, None, d["beta"], w.T)
    else:
        X = qs.Inputs(d["q"], d["k"], d["v"], None, s_code, s_lut, d["beta"], w.T)
    S = torch.zeros((w.B, w.H, w.dk, w.dv), dtype=torch.float32, device="cuda")
    o = torch.zeros((w.B, w.T, w.H, w.dv), dtype=torch.float32, device="cuda")
    qs.qstate_scan_fp32(cfg, S, X, 0, w.T, o)
    qs.qstate_check()
    return o.cpu().numpy().astype(np.float64)


def test_log_uniform_gates_keep_readouts(qs, orc):
    """Sec. 3, "Decay-gate quantization": the readout error that the library's log-uniform
    decay-rate quantiser costs the unquantised state (KDA inputs, rates s = softplus(N(-2, 1))
    drawn every token), against the recurrence on the exact rates: smaller with more levels, and
    equal to the error computed with the oracle's quantiser and its FP64 recurrence."""
    w = synth.scaled(synth.WORKLOADS["kda_decode"], B=2, H=2, T=256, gate_bits=0)
    inp = synth.host_inputs(w)
    nchan = w.H * w.dk
    ref = _fp32_readouts_with_rates(qs, w, inp)
    den = np.sum(ref ** 2)
    s_dev = torch.from_numpy(inp["s"]).cuda()
    errs = {}
    for g in (2, 4):
        cfg = qs.Config.from_workload(w, gate_bits=g)
        L = 1 << g
        codes = torch.zeros(s_dev.shape, dtype=torch.uint8, device="cuda")
        lut = torch.zeros(nchan * L, dtype=torch.float32, device="cuda")
        thr = torch.zeros(nchan * (L - 1), dtype=torch.float32, device="cuda")
        qs.qstate_quant_decay(cfg, s_dev, codes, lut, thr)
        o = _fp32_readouts_with_rates(qs, w, inp, codes, lut, g)
        errs[f"log g={g}"] = float(np.sum((o - ref) ** 2) / den)
    print("relative readout MSE:", ", ".join(f"{k} {v:.4e}" for k, v in errs.items()))
    assert errs["log g=4"] < 0.1 * errs["log g=2"], errs
    # the same error from the oracle's quantiser and FP64 recurrence
    c_ref, l_ref, _ = orc.quant_decay(inp["s"], nchan, 2)
    cfgo = orc.Cfg.from_workload(w)
    sq = l_ref[np.arange(nchan)[None, None, :], c_ref.reshape(w.B, w.T, nchan)].reshape(inp["s"].shape)
    x = dict(inp)
    x["s"] = sq.astype(np.float32)
    e = 0.0
    ref64 = np.zeros_like(ref)
    for b in range(w.B):
        for h in range(w.H):
            o64, _ = orc.recur(np.zeros((w.dk, w.dv)), *orc.expand_inputs(cfgo, x, b, h), dtype=np.float64)
            r64, _ = orc.recur(np.zeros((w.dk, w.dv)), *orc.expand_inputs(cfgo, inp, b, h), dtype=np.float64)
            e += np.sum((o64 - r64) ** 2)
            ref64[b, :, h] = r64
    e_orc = e / np.sum(ref64 ** 2)
    print(f"oracle, log g=2: {e_orc:.4e}")
    assert abs(errs["log g=2"] - e_orc) <= 0.01 * e_orc, (errs["log g=2"], e_orc)
