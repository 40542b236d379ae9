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
