"""CPU checks of the C ABI: the library builds and loads, exports every function declared in
include/qstate.h, and its host-only calls (validation, sizes, bit accounting) behave.  No
kernel is launched."""
import ctypes as ct
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    from paper_2609_30950_gb300 import build
    import paper_2609_30950_gb300 as q
    build.build()
    return q.load()


def _declared():
    src = open(os.path.join(ROOT, "include", "qstate.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(qstate_[a-z0-9_]+)\s*\(", src)))


def test_exports_every_declared_symbol(lib):
    names = _declared()
    assert len(names) >= 14
    for name in names:
        assert hasattr(lib, name), name
        assert ct.cast(getattr(lib, name), ct.c_void_p).value


def test_binding_names_cover_header():
    import paper_2609_30950_gb300 as q
    assert sorted(q.EXPORTS) == _declared()


def test_validation_and_sizes(lib):
    import paper_2609_30950_gb300 as q
    import synth
    for name, w in synth.WORKLOADS.items():
        cfg = q.Config.from_workload(w)
        q.validate(cfg)
        assert q.region_bytes(cfg) == w.H * w.dk * w.dv * w.bbar // 8
    bad = [dict(dk=96), dict(bmax=17), dict(bmin=5, bbar_num=4), dict(group_heads=3),
           dict(C=0), dict(gate_bits=9), dict(unit_kind=q.UNIT_HEAD, decay_kind=q.DECAY_ROW)]
    for kw in bad:
        base = dict(B=2, H=4, dk=128, dv=128)
        base.update(kw)
        cfg = q.Config(**base)
        with pytest.raises(q.QstateError) as e:
            q.validate(cfg)
        assert e.value.code in (q.QSTATE_EINVAL, q.QSTATE_EBUDGET)
    with pytest.raises(q.QstateError) as e:
        q.validate(q.Config(B=1, H=2, dk=64, dv=64, bbar_num=4, bmin=5, bmax=8))
    assert e.value.code == q.QSTATE_EBUDGET


def test_bits_per_element_agrees_with_oracle(lib, orc):
    import paper_2609_30950_gb300 as q
    import synth
    for w in synth.WORKLOADS.values():
        a = q.bits_per_element(q.Config.from_workload(w))
        b = orc.bits_per_element(orc.Cfg.from_workload(w))
        assert a == b


def test_calls_reject_null_pointers_without_launching(lib):
    import paper_2609_30950_gb300 as q
    cfg = q.Config(B=1, H=1, dk=64, dv=64, bbar_num=2, bmin=1, bmax=16).c()
    assert lib.qstate_pack(ct.byref(cfg), None, None, None, None) == q.QSTATE_EINVAL
    assert b"null" in lib.qstate_last_error()


def test_chunked_form_configuration_limits(lib):
    """The chunked form (interval_form = 1) is for the row unit at dk = dv = 128 with the
    delta rule or no erasure; anything else is rejected before a launch."""
    import paper_2609_30950_gb300 as q
    q.validate(q.Config(B=1, H=2, dk=128, dv=128, interval_form=q.FORM_CHUNK))
    q.validate(q.Config(B=1, H=2, dk=128, dv=128, erase_kind=q.ERASE_NONE, decay_kind=q.DECAY_HEAD,
                        interval_form=q.FORM_CHUNK))
    for kw in (dict(dk=64, dv=64), dict(unit_kind=q.UNIT_HEAD, decay_kind=q.DECAY_HEAD),
               dict(erase_kind=q.ERASE_GENERAL), dict(interval_form=2)):
        base = dict(B=1, H=2, dk=128, dv=128, interval_form=q.FORM_CHUNK)
        base.update(kw)
        with pytest.raises(q.QstateError) as e:
            q.validate(q.Config(**base))
        assert e.value.code == q.QSTATE_EINVAL


def test_scan_partition_setter_checks_its_range(lib):
    # no launch: the setter only records the request
    from paper_2609_30950_gb300 import QSTATE_EINVAL, QSTATE_OK
    assert lib.qstate_set_scan_partitions(9) == QSTATE_EINVAL
    assert lib.qstate_set_scan_partitions(-1) == QSTATE_EINVAL
    for n in (8, 1, 0):
        assert lib.qstate_set_scan_partitions(n) == QSTATE_OK


def _part_count(lib, w, parts, form=0, s_code=False, beta=True):
    """qstate_scan_partition_count on host-only arguments: placeholder device addresses (the
    call only checks them for NULL and never dereferences them)."""
    import paper_2609_30950_gb300 as q
    cfg = q.Config.from_workload(w, interval_form=form).c()
    A = 1 << 20
    x = q._Inputs(A, A, A, None if s_code else A, A if s_code else None, A if s_code else None,
                  A if beta else None, w.T, None, None)
    st = q._Stats(A, A, A)
    assert lib.qstate_set_scan_partitions(parts) == 0
    try:
        return lib.qstate_scan_partition_count(ct.byref(cfg), ct.byref(x), ct.byref(st))
    finally:
        lib.qstate_set_scan_partitions(0)


def test_scan_partition_count_rule(lib):
    """Batch partitions of a scan: 4 in the token form and 2 in the chunked form by default, at
    most one per batch element, and fewer where a partition would start off a 16-byte boundary
    in any array."""
    import synth
    kda = synth.scaled(synth.WORKLOADS["kda_decode"], B=16, H=8, T=48)
    assert _part_count(lib, kda, 0, s_code=True) == 4
    assert _part_count(lib, kda, 0, form=1) == 2
    assert _part_count(lib, kda, 8) == 8
    assert _part_count(lib, synth.scaled(kda, B=3), 8) == 3
    assert _part_count(lib, synth.scaled(kda, B=1), 0) == 1
    assert _part_count(lib, kda, 1) == 1
    # head unit with H = 3: 3 width bytes per batch element, so a partition may start only at a
    # multiple of 16 elements; with B = 32 that leaves the split at element 16
    gdn = synth.scaled(synth.WORKLOADS["gdn_decode"], B=32, H=3, T=16)
    assert _part_count(lib, gdn, 4) == 2
    assert _part_count(lib, gdn, 8) == 2
    # per-head rates of an odd token count: 4 T H bytes per element, T H = 3 x 17
    gdn_odd = synth.scaled(synth.WORKLOADS["gdn_decode"], B=4, H=16, T=17)
    assert _part_count(lib, gdn_odd, 4) == 4          # 4 x 17 x 16 = 1088: aligned
    kda_odd = synth.scaled(kda, B=4, T=17)            # rate codes: T H dk bytes, aligned
    assert _part_count(lib, kda_odd, 4, s_code=True) == 4
    # an invalid configuration or missing statistics: 0
    import paper_2609_30950_gb300 as q
    cfg = q.Config.from_workload(kda).c()
    x = q._Inputs(1 << 20, 1 << 20, 1 << 20, 1 << 20, None, None, 1 << 20, kda.T, None, None)
    assert lib.qstate_scan_partition_count(ct.byref(cfg), ct.byref(x), None) == 0
    bad = q.Config.from_workload(kda, C=0).c()
    st = q._Stats(1 << 20, 1 << 20, 1 << 20)
    assert lib.qstate_scan_partition_count(ct.byref(bad), ct.byref(x), ct.byref(st)) == 0
