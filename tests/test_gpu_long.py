"""Full-length lockstep on the benchmark layer shapes (GPU): every write-back of the whole
sequence, all heads, four batch elements (KDA decode, Mamba-2) or two (Gated DeltaNet, KDA
prefill).

* KDA decode: 1024 per-token write-backs, log-coded rates (H = 32, 128 x 128, 4 bits).
* Gated DeltaNet: 2048 per-token write-backs (head unit, H = 16).
* Mamba-2: 2048 per-token write-backs (H = 64, 128 x 64, 6 bits).
* KDA prefill: 8192 tokens in chunked form on the tensor cores, 128 write-backs of C = 64.

Eq. (1) with the EMA statistics of Sec. 3 (span 64) and lagged widths is stateful over
hundreds of tokens, so these runs check that the kernels' EMAs, ranges, widths and states keep
tracking the oracle over the whole sequence.  At every write-back the oracle's packed state is
handed to the GPU (lockstep): readouts within 1e-5 normwise over each token's heads (1e-3 per
vector), codes >= 99.99 % identical and within one step, statistics within 1e-5, the next widths
bit-exact through the allocation kernel.

Afterwards the GPU runs the same sequence free (its own state throughout) and the divergence
of its readouts from the oracle's free run is printed: off-by-one codes inject step-sized noise
that the recurrence carries, so this comparison is reported, not bounded (Sec. 2, "Accumulated
readout error").  Beside it, both free runs are compared with the unquantised FP32 recurrence
on the same (decoded) rates: the quantised state's own readout error, which the two should
share.
"""
from concurrent.futures import ThreadPoolExecutor

import numpy as np
import pytest

import synth
from parity import host
from test_gpu_parity import _dev_inputs, _lockstep

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")

# name -> (log-coded rates, interval form, batch elements)
LONG = {
    "kda_decode": (True, 0, 4),
    "gdn_decode": (False, 0, 2),
    "mamba2_decode": (False, 0, 4),
    "kda_prefill": (False, 1, 2),
}


@pytest.mark.parametrize("name", list(LONG))
def test_full_length_lockstep(qs, orc, name):
    log_decay, form, nb = LONG[name]
    w = synth.scaled(synth.WORKLOADS[name], B=nb)
    inp = synth.host_inputs(w)
    # the oracle's OpenMP build (bit-identical to the plain build, pinned on the CPU) keeps the
    # host side of four full-length batch elements within minutes
    rep, o_orc = _lockstep(qs, orc, w, log_decay=log_decay, interval_form=form,
                           sample_b=tuple(range(nb)), inputs=inp, oracle_parallel=True)
    assert len(rep) == nb * ((w.T + w.C - 1) // w.C)
    worst = max(r["rel_o"] for r in rep)
    worst_v = max(r["rel_o_vec"] for r in rep)
    agree = min(r["code_agree"] for r in rep)
    ties = sum(r["fidx_diff"] for r in rep)
    scale_ulps = sum(r["scale_diff"] for r in rep)
    print(f"\n{name}: T = {w.T}, {len(rep) // nb} write-backs x {nb} batch elements in lockstep: worst "
          f"rel readout {worst:.2e} per token ({worst_v:.2e} per vector), min code agreement {agree:.6f}, near-tie factor differences "
          f"{ties}, one-ulp scale differences {scale_ulps}")

    # the same sequence run free on the GPU, against the oracle's free run (reported)
    cfgq = qs.Config.from_workload(w, interval_form=form)
    s_code = s_lut = None
    if log_decay:
        nchan = w.H * w.dk if w.per_row_decay else w.H
        s_code, s_lut, _ = orc.quant_decay(inp["s"], nchan, w.gate_bits)
    X, _ = _dev_inputs(w, inp, qs, s_code, s_lut)
    A, Bs = qs.new_state(cfgq), qs.new_state(cfgq)
    qs.qstate_init(cfgq, A, Bs)
    st = qs.new_stats(cfgq)
    o = torch.zeros((w.B, w.T, w.H, w.dv), dtype=torch.float32, device="cuda")
    qs.qstate_scan(cfgq, A, Bs, X, 0, w.T, 0, o, st)
    qs.qstate_check()
    og = host(o, np.float64)
    ref = np.concatenate([o_orc[b] for b in range(nb)], axis=0).astype(np.float64)
    num = np.linalg.norm(og - ref, axis=-1)
    den = np.maximum(np.linalg.norm(ref, axis=-1), 1e-30)
    e = num / den
    assert np.isfinite(og).all()
    q = w.T // 4
    print(f"{name}: free-running GPU vs free-running oracle, relative readout error per (b, t, h): "
          f"median {np.median(e):.2e}, mean {e.mean():.2e}, max {e.max():.2e}; mean over the first / "
          f"last quarter of tokens {e[:, :q].mean():.2e} / {e[:, -q:].mean():.2e}; relative "
          f"readout MSE {np.sum(num ** 2) / np.sum(den ** 2):.2e}")

    # the unquantised FP32 recurrence (Eq. 1) on the rates both runs used
    cfgo = orc.Cfg.from_workload(w)
    ex = dict(inp)
    if log_decay:
        chan = np.arange(w.H * w.dk).reshape(w.H, w.dk) if w.per_row_decay else np.arange(w.H)
        ex["s"] = s_lut[chan, s_code.astype(np.int64)].astype(np.float32)
    pairs = [(b, h) for b in range(w.B) for h in range(w.H)]

    def exact(bh):
        b, h = bh
        o32, _ = orc.recur(np.zeros((w.dk, w.dv)), *orc.expand_inputs(cfgo, ex, b, h), dtype=np.float32)
        return o32
    with ThreadPoolExecutor(max_workers=8) as pool:
        outs = list(pool.map(exact, pairs))
    o_ex = np.zeros_like(ref)
    for (b, h), o32 in zip(pairs, outs):
        o_ex[b, :, h] = o32
    mse = lambda a: float(np.sum((a - o_ex) ** 2) / np.sum(o_ex ** 2))
    print(f"{name}: relative readout MSE against the unquantised FP32 recurrence: GPU free run "
          f"{mse(og):.3e}, oracle free run {mse(ref):.3e}")
