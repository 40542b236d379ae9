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


def _gpu_rel_mse(qs, w, weight_kind, o_ref):
    cfg = qs.Config.from_workload(w, weight_kind=weight_kind)
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
CASES = [(64, 2, 1, 8, 512, 0.5), (16, 2, 1, 8, 512, 0.5), (1, 4, 0, 8, 256, 0.4)]


@pytest.mark.parametrize("C,bbar,bmin,bmax,T,ratio", CASES)
def test_allocation_lowers_readout_error(qs, orc, C, bbar, bmin, bmax, T, ratio):
    W = _workload(C, bbar, bmin, bmax, T)
    o_ref = _gpu_fp32_readouts(qs, W)
    errs = {name: _gpu_rel_mse(qs, W, kind, o_ref)
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
