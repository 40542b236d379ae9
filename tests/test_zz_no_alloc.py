"""qstate_quant_decay_noalloc against qstate_quant_decay (GPU).

The variant keeps the quantiser's thresholds in a fixed array inside the library instead of a
caller buffer; its codes and levels must be those of the entry point with a caller buffer,
bit for bit, on consecutive calls (the second call sees the first call's leftovers in the
array).  This file is collected last so that it also runs after every other GPU test.
"""
import numpy as np
import pytest
import torch

import synth

pytestmark = pytest.mark.gpu

CASES = [("tiny_kda", 2), ("kda_decode", 4), ("gdn_decode", 3), ("mamba2_decode", 8)]


def _quantise(qs, w, noalloc):
    cfg = qs.Config.from_workload(w)
    s = torch.from_numpy(synth.host_inputs(w)["s"]).cuda()
    nchan = w.H * w.dk if w.per_row_decay else w.H
    L = 2 ** w.gate_bits
    codes = torch.full(s.shape, 0xAB, dtype=torch.uint8, device="cuda")
    lut = torch.full((nchan * L,), float("nan"), dtype=torch.float32, device="cuda")
    if noalloc:
        qs.qstate_quant_decay_noalloc(cfg, s, codes, lut)
    else:
        thr = torch.zeros(nchan * (L - 1), dtype=torch.float32, device="cuda")
        qs.qstate_quant_decay(cfg, s, codes, lut, thr)
    qs.qstate_check()
    return codes.cpu().numpy(), lut.cpu().numpy()


@pytest.mark.parametrize("name,g", CASES)
def test_noalloc_matches_entry_point_on_consecutive_calls(qs, name, g):
    base = synth.WORKLOADS[name]
    for call in range(2):
        w = synth.scaled(base, B=min(base.B, 4), T=37, gate_bits=g, seed=base.seed + 17 * call)
        c_ref, l_ref = _quantise(qs, w, noalloc=False)
        c_new, l_new = _quantise(qs, w, noalloc=True)
        assert np.array_equal(c_new, c_ref), f"{name} call {call}: codes differ"
        assert np.array_equal(l_new.view(np.uint32), l_ref.view(np.uint32)), \
            f"{name} call {call}: levels differ"


def test_noalloc_after_a_larger_table(qs):
    # a large table (4096 channels x 15 thresholds) then a small one: the small call must
    # read only the entries it wrote itself
    big = synth.scaled(synth.WORKLOADS["kda_decode"], B=2, T=9, gate_bits=4)
    small = synth.scaled(synth.WORKLOADS["gdn_decode"], B=3, T=11, gate_bits=2)
    for w in (big, small, big):
        c_ref, l_ref = _quantise(qs, w, noalloc=False)
        c_new, l_new = _quantise(qs, w, noalloc=True)
        assert np.array_equal(c_new, c_ref)
        assert np.array_equal(l_new.view(np.uint32), l_ref.view(np.uint32))


def test_noalloc_at_the_largest_table_that_fits(qs):
    # 257 heads x 255 thresholds (per-head rates, gate_bits = 8) = 65535: the largest table the
    # configuration limits allow at or below the 65536-entry array (65536 itself would need
    # 65536 channels at one threshold each); bit for bit against the caller-buffer entry point,
    # twice in a row
    for call in range(2):
        w = synth.scaled(synth.WORKLOADS["gdn_decode"], B=2, H=257, T=5, gate_bits=8, seed=31 + call)
        assert w.H * (2 ** w.gate_bits - 1) == 65535
        c_ref, l_ref = _quantise(qs, w, noalloc=False)
        c_new, l_new = _quantise(qs, w, noalloc=True)
        assert np.array_equal(c_new, c_ref)
        assert np.array_equal(l_new.view(np.uint32), l_ref.view(np.uint32))


@pytest.mark.parametrize("H", [258, 1024])
def test_noalloc_rejects_one_channel_over(qs, H):
    # 258 heads x 255 = 65790 thresholds: one channel past the array
    w = synth.scaled(synth.WORKLOADS["gdn_decode"], B=1, H=H, T=2, gate_bits=8)
    cfg = qs.Config.from_workload(w)
    s = torch.ones((1, 2, H), dtype=torch.float32, device="cuda")
    codes = torch.full(s.shape, 7, dtype=torch.uint8, device="cuda")
    lut = torch.zeros(H * 256, dtype=torch.float32, device="cuda")
    with pytest.raises(qs.QstateError) as e:
        qs.qstate_quant_decay_noalloc(cfg, s, codes, lut)
    assert e.value.code == qs.QSTATE_EINVAL
    qs.qstate_check()
    assert bool((codes == 7).all()) and bool((lut == 0).all())


def test_noalloc_rejects_tables_above_its_maximum(qs):
    # 4096 channels x (2^5 - 1) = 126976 thresholds > 65536
    w = synth.scaled(synth.WORKLOADS["kda_decode"], B=1, T=2, gate_bits=5)
    cfg = qs.Config.from_workload(w)
    s = torch.ones((1, 2, w.H, w.dk), dtype=torch.float32, device="cuda")
    codes = torch.full(s.shape, 7, dtype=torch.uint8, device="cuda")
    lut = torch.zeros(w.H * w.dk * 32, dtype=torch.float32, device="cuda")
    with pytest.raises(qs.QstateError) as e:
        qs.qstate_quant_decay_noalloc(cfg, s, codes, lut)
    assert e.value.code == qs.QSTATE_EINVAL
    assert "65536" in str(e.value)
    qs.qstate_check()
    assert bool((codes == 7).all()) and bool((lut == 0).all())   # nothing was launched
