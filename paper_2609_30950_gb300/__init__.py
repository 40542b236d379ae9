"""Python binding of libqstate (the C ABI in include/qstate.h).

Argument marshalling only: every step of the hot path runs in the CUDA library.  Tensors are
torch tensors on a CUDA device (torch supplies device memory and streams); the library is
loaded from this package's in-tree build and there is no fallback -- without the compiled
library every call raises.
"""
from __future__ import annotations

import ctypes as ct
import os
from dataclasses import dataclass, field

from . import build as _build

QSTATE_OK, QSTATE_EINVAL, QSTATE_EBUDGET, QSTATE_ECUDA, QSTATE_EDEVICE, QSTATE_ETIMEOUT = range(6)
DECAY_ROW, DECAY_HEAD = 0, 1
ERASE_DELTA, ERASE_NONE, ERASE_GENERAL = 0, 1, 2
ALLOC_LAGGED, ALLOC_CURRENT = 0, 1
FORM_TOKEN, FORM_CHUNK = 0, 1
UNIT_ROW, UNIT_HEAD = 0, 1
# allocation weights (Eq. 3 and the alternatives of Table 1; see include/qstate.h)
(WEIGHT_OURS, WEIGHT_RANGE, WEIGHT_GAMMA_RAW, WEIGHT_NRANGE, WEIGHT_PERSIST, WEIGHT_WBFACTOR,
 WEIGHT_NOERASE, WEIGHT_SHUFFLE, WEIGHT_UNIFORM) = range(9)


class QstateError(RuntimeError):
    def __init__(self, code: int, msg: str):
        super().__init__(f"qstate error {code}: {msg}")
        self.code = code


class _Cfg(ct.Structure):
    _fields_ = [("B", ct.c_int32), ("H", ct.c_int32), ("dk", ct.c_int32), ("dv", ct.c_int32),
                ("decay_kind", ct.c_int32), ("erase_kind", ct.c_int32),
                ("unit_kind", ct.c_int32), ("group_heads", ct.c_int32),
                ("bbar_num", ct.c_int32), ("bbar_den", ct.c_int32), ("bmin", ct.c_int32),
                ("bmax", ct.c_int32), ("C", ct.c_int32), ("fit_every", ct.c_int32),
                ("ema_span", ct.c_float), ("gate_bits", ct.c_int32),
                ("weight_kind", ct.c_int32), ("alloc_mode", ct.c_int32),
                ("interval_form", ct.c_int32)]


class _Buf(ct.Structure):
    _fields_ = [("payload", ct.c_void_p), ("scales", ct.c_void_p), ("widths", ct.c_void_p),
                ("head_off", ct.c_void_p), ("fidx", ct.c_void_p)]


class _Stats(ct.Structure):
    _fields_ = [("ema_s", ct.c_void_p), ("ema_r", ct.c_void_p), ("range", ct.c_void_p)]


class _Inputs(ct.Structure):
    _fields_ = [("q", ct.c_void_p), ("k", ct.c_void_p), ("v", ct.c_void_p), ("s", ct.c_void_p),
                ("s_code", ct.c_void_p), ("s_lut", ct.c_void_p), ("beta", ct.c_void_p),
                ("T", ct.c_int32), ("a", ct.c_void_p), ("w", ct.c_void_p)]


EXPORTS = ["qstate_validate", "qstate_region_bytes", "qstate_units", "qstate_scale_groups",
           "qstate_bits_per_element", "qstate_init", "qstate_alloc_bits", "qstate_pack",
           "qstate_unpack", "qstate_quant_decay", "qstate_quant_decay_noalloc", "qstate_step",
           "qstate_scan", "qstate_scan_host",
           "qstate_scan_fp32", "qstate_check", "qstate_set_wait_limit", "qstate_set_scan_partitions",
           "qstate_scan_partition_count", "qstate_last_error"]

_lib = None


def library_path() -> str:
    return _build.LIB


def load(path: str | None = None, build_if_missing: bool = False):
    """Load libqstate.so (build it first if asked).  Raises if it is missing."""
    global _lib
    if _lib is not None:
        return _lib
    path = path or _build.LIB
    if not os.path.exists(path):
        if not build_if_missing:
            raise QstateError(QSTATE_ECUDA, f"CUDA library not built: {path} (run build())")
        _build.build()
    L = ct.CDLL(path)
    P, PC = ct.c_void_p, ct.POINTER(_Cfg)
    L.qstate_validate.argtypes = [PC]
    L.qstate_region_bytes.argtypes = [PC]
    L.qstate_region_bytes.restype = ct.c_size_t
    L.qstate_units.argtypes = [PC]
    L.qstate_units.restype = ct.c_size_t
    L.qstate_scale_groups.argtypes = [PC]
    L.qstate_scale_groups.restype = ct.c_size_t
    L.qstate_bits_per_element.argtypes = [PC]
    L.qstate_bits_per_element.restype = ct.c_double
    L.qstate_init.argtypes = [PC, ct.POINTER(_Buf), ct.POINTER(_Buf), P]
    L.qstate_alloc_bits.argtypes = [PC, ct.POINTER(_Stats), P, P, P]
    L.qstate_pack.argtypes = [PC, P, ct.POINTER(_Buf), P, P]
    L.qstate_unpack.argtypes = [PC, ct.POINTER(_Buf), P, P]
    L.qstate_quant_decay.argtypes = [PC, P, ct.c_int32, P, P, P, P]
    L.qstate_quant_decay_noalloc.argtypes = [PC, P, ct.c_int32, P, P, P]
    L.qstate_step.argtypes = [PC, ct.POINTER(_Buf), ct.POINTER(_Buf), ct.POINTER(_Inputs),
                              ct.c_int32, ct.c_int32, ct.c_int32, P, ct.POINTER(_Stats), P]
    L.qstate_scan.argtypes = [PC, ct.POINTER(_Buf), ct.POINTER(_Buf), ct.POINTER(_Inputs),
                              ct.c_int32, ct.c_int32, ct.c_int32, P, ct.POINTER(_Stats),
                              ct.POINTER(ct.c_int32), P]
    L.qstate_scan_host.argtypes = [PC, ct.POINTER(_Buf), ct.POINTER(_Buf), ct.POINTER(_Inputs),
                                   ct.POINTER(_Inputs), ct.c_int32, ct.c_int32, ct.c_int32, P, P,
                                   ct.POINTER(_Stats), ct.c_int32, ct.POINTER(ct.c_int32), P, P]
    L.qstate_scan_fp32.argtypes = [PC, P, ct.POINTER(_Inputs), ct.c_int32, ct.c_int32, P, P]
    L.qstate_check.argtypes = [P]
    L.qstate_set_wait_limit.argtypes = [ct.c_int32]
    L.qstate_set_scan_partitions.argtypes = [ct.c_int32]
    L.qstate_scan_partition_count.argtypes = [ct.c_void_p, ct.c_void_p, ct.c_void_p]
    L.qstate_last_error.restype = ct.c_char_p
    for name in EXPORTS:
        if name not in ("qstate_region_bytes", "qstate_units", "qstate_scale_groups",
                        "qstate_bits_per_element", "qstate_last_error"):
            getattr(L, name).restype = ct.c_int
    _lib = L
    return L


def _lib_or_raise():
    return _lib if _lib is not None else load()


def _check(rc: int):
    if rc != QSTATE_OK:
        raise QstateError(rc, _lib_or_raise().qstate_last_error().decode())


def _ptr(t):
    if t is None:
        return None
    if not t.is_cuda:
        raise ValueError("tensor must live on a CUDA device")
    if not t.is_contiguous():
        raise ValueError("tensor must be contiguous")
    return ct.c_void_p(t.data_ptr())


def _stream(stream):
    import torch
    s = stream if stream is not None else torch.cuda.current_stream()
    return ct.c_void_p(s.cuda_stream)


@dataclass
class Config:
    """Method configuration (mirrors ``qstate_cfg``)."""
    B: int
    H: int
    dk: int
    dv: int
    decay_kind: int = DECAY_ROW
    erase_kind: int = ERASE_DELTA
    unit_kind: int = UNIT_ROW
    group_heads: int = 1
    bbar_num: int = 4
    bbar_den: int = 1
    bmin: int = 1
    bmax: int = 8
    C: int = 1
    fit_every: int = 1
    ema_span: float = 64.0
    gate_bits: int = 0
    weight_kind: int = 0
    alloc_mode: int = 0
    interval_form: int = 0

    def c(self) -> _Cfg:
        return _Cfg(*[getattr(self, f) for f, _ in _Cfg._fields_])

    @classmethod
    def from_workload(cls, w, **over) -> "Config":
        kw = dict(B=w.B, H=w.H, dk=w.dk, dv=w.dv,
                  decay_kind=DECAY_ROW if w.per_row_decay else DECAY_HEAD,
                  erase_kind=(ERASE_GENERAL if getattr(w, "general", False)
                            else ERASE_DELTA if w.erase else ERASE_NONE),
                  unit_kind=UNIT_ROW if w.unit == "row" else UNIT_HEAD,
                  group_heads=w.group_heads, bbar_num=w.bbar, bbar_den=1, bmin=w.bmin,
                  bmax=w.bmax, C=w.C, gate_bits=w.gate_bits)
        kw.update(over)
        return cls(**kw)

    @property
    def units(self) -> int:
        return self.H * self.dk if self.unit_kind == UNIT_ROW else self.H

    @property
    def scale_groups(self) -> int:
        return self.H * self.dk if self.unit_kind == UNIT_ROW else self.H * (self.dk // 32) * self.dv


def validate(cfg: Config) -> None:
    c = cfg.c()
    _check(_lib_or_raise().qstate_validate(ct.byref(c)))


def region_bytes(cfg: Config) -> int:
    validate(cfg)
    c = cfg.c()
    return int(_lib_or_raise().qstate_region_bytes(ct.byref(c)))


def bits_per_element(cfg: Config) -> float:
    validate(cfg)
    c = cfg.c()
    return float(_lib_or_raise().qstate_bits_per_element(ct.byref(c)))


@dataclass
class State:
    """One packed state (device tensors, caller-owned)."""
    payload: object
    scales: object
    widths: object
    head_off: object
    fidx: object

    def c(self) -> _Buf:
        return _Buf(*(_ptr(t) for t in (self.payload, self.scales, self.widths, self.head_off,
                                          self.fidx)))


def new_state(cfg: Config, device="cuda") -> State:
    import torch
    rb = region_bytes(cfg)
    return State(torch.zeros(cfg.B * rb, dtype=torch.uint8, device=device),
                 torch.zeros(cfg.B * cfg.scale_groups, dtype=torch.int16, device=device),
                 torch.zeros(cfg.B * cfg.units, dtype=torch.uint8, device=device),
                 torch.zeros(cfg.B * cfg.H, dtype=torch.int32, device=device),
                 torch.full((cfg.B * cfg.scale_groups,), 15, dtype=torch.uint8, device=device))


@dataclass
class Stats:
    ema_s: object
    ema_r: object
    range: object

    def c(self) -> _Stats:
        return _Stats(_ptr(self.ema_s), _ptr(self.ema_r), _ptr(self.range))


def new_stats(cfg: Config, device="cuda") -> Stats:
    import torch
    n = cfg.B * cfg.units
    return Stats(*(torch.zeros(n, dtype=torch.float32, device=device) for _ in range(3)))


@dataclass
class Inputs:
    q: object
    k: object
    v: object
    s: object = None
    s_code: object = None
    s_lut: object = None
    beta: object = None
    T: int = field(default=0)
    a: object = None
    w: object = None

    def c(self) -> _Inputs:
        T = self.T or int(self.q.shape[1])
        return _Inputs(_ptr(self.q), _ptr(self.k), _ptr(self.v), _ptr(self.s), _ptr(self.s_code),
                       _ptr(self.s_lut), _ptr(self.beta), T, _ptr(self.a), _ptr(self.w))


def qstate_init(cfg: Config, a: State, b: State, stream=None) -> None:
    c, ba, bb = cfg.c(), a.c(), b.c()
    _check(_lib_or_raise().qstate_init(ct.byref(c), ct.byref(ba), ct.byref(bb), _stream(stream)))


def qstate_alloc_bits(cfg: Config, stats: Stats, widths_out, head_off_out, stream=None) -> None:
    c, st = cfg.c(), stats.c()
    _check(_lib_or_raise().qstate_alloc_bits(ct.byref(c), ct.byref(st), _ptr(widths_out),
                                             _ptr(head_off_out), _stream(stream)))


def qstate_pack(cfg: Config, S, out: State, range_out=None, stream=None) -> None:
    c, bo = cfg.c(), out.c()
    _check(_lib_or_raise().qstate_pack(ct.byref(c), _ptr(S), ct.byref(bo), _ptr(range_out),
                                       _stream(stream)))


def qstate_unpack(cfg: Config, src: State, S_out, stream=None) -> None:
    c, bi = cfg.c(), src.c()
    _check(_lib_or_raise().qstate_unpack(ct.byref(c), ct.byref(bi), _ptr(S_out), _stream(stream)))


def qstate_quant_decay(cfg: Config, s, code_out, lut_out, thr_out, stream=None) -> None:
    c = cfg.c()
    _check(_lib_or_raise().qstate_quant_decay(ct.byref(c), _ptr(s), int(s.shape[1]), _ptr(code_out),
                                              _ptr(lut_out), _ptr(thr_out), _stream(stream)))


def qstate_quant_decay_noalloc(cfg: Config, s, code_out, lut_out, stream=None) -> None:
    """qstate_quant_decay without a threshold buffer (see include/qstate.h)."""
    c = cfg.c()
    _check(_lib_or_raise().qstate_quant_decay_noalloc(ct.byref(c), _ptr(s), int(s.shape[1]),
                                                      _ptr(code_out), _ptr(lut_out),
                                                      _stream(stream)))


def qstate_step(cfg: Config, src: State, dst: State, x: Inputs, t_begin: int, t_end: int,
                w_index: int, o, stats: Stats, stream=None) -> None:
    c, bi, bo, xi, st = cfg.c(), src.c(), dst.c(), x.c(), stats.c()
    _check(_lib_or_raise().qstate_step(ct.byref(c), ct.byref(bi), ct.byref(bo), ct.byref(xi),
                                       t_begin, t_end, w_index, _ptr(o), ct.byref(st),
                                       _stream(stream)))


def qstate_scan(cfg: Config, ping: State, pong: State, x: Inputs, t_begin: int, t_end: int,
                w_index0: int, o, stats: Stats, stream=None) -> bool:
    """Returns True if the final state is in ``pong``."""
    c, bi, bo, xi, st = cfg.c(), ping.c(), pong.c(), x.c(), stats.c()
    flag = ct.c_int32(0)
    _check(_lib_or_raise().qstate_scan(ct.byref(c), ct.byref(bi), ct.byref(bo), ct.byref(xi),
                                       t_begin, t_end, w_index0, _ptr(o), ct.byref(st),
                                       ct.byref(flag), _stream(stream)))
    return bool(flag.value)


def _hptr(t):
    """Pointer of a host (CPU) tensor; pinned memory keeps the copies asynchronous."""
    if t is None:
        return None
    if t.is_cuda or not t.is_contiguous():
        raise ValueError("host tensor must be a contiguous CPU tensor")
    return ct.c_void_p(t.data_ptr())


def qstate_scan_host(cfg: Config, ping: State, pong: State, x_host: Inputs, x_dev: Inputs,
                     t_begin: int, t_end: int, w_index0: int, o_host, o_dev, stats: Stats,
                     chunk: int, stream, copy_stream) -> bool:
    """qstate_scan with inputs staged from host tensors chunk by chunk (see include/qstate.h).
    Returns True if the final state is in ``pong``."""
    c, bi, bo, st = cfg.c(), ping.c(), pong.c(), stats.c()
    xh = _Inputs(*(_hptr(getattr(x_host, n)) for n in ("q", "k", "v", "s", "s_code", "s_lut", "beta")),
                 x_host.T or int(x_host.q.shape[1]), _hptr(x_host.a), _hptr(x_host.w))
    xd = x_dev.c()
    flag = ct.c_int32(0)
    _check(_lib_or_raise().qstate_scan_host(ct.byref(c), ct.byref(bi), ct.byref(bo), ct.byref(xh),
                                            ct.byref(xd), t_begin, t_end, w_index0, _hptr(o_host),
                                            _ptr(o_dev), ct.byref(st), chunk, ct.byref(flag),
                                            ct.c_void_p(stream.cuda_stream),
                                            ct.c_void_p(copy_stream.cuda_stream)))
    return bool(flag.value)


def qstate_scan_fp32(cfg: Config, S, x: Inputs, t_begin: int, t_end: int, o, stream=None) -> None:
    c, xi = cfg.c(), x.c()
    _check(_lib_or_raise().qstate_scan_fp32(ct.byref(c), _ptr(S), ct.byref(xi), t_begin, t_end,
                                            _ptr(o), _stream(stream)))


def qstate_check(stream=None) -> None:
    _check(_lib_or_raise().qstate_check(_stream(stream)))


def qstate_set_wait_limit(polls: int) -> None:
    """Limit of the chunked form's waits for its tensor-core products in later calls (polls;
    0 gives up at once, negative restores the default)."""
    _check(_lib_or_raise().qstate_set_wait_limit(int(polls)))


def qstate_set_scan_partitions(n: int) -> None:
    """Batch partitions of later scans, each on its own stream (1..8; 0 chooses per
    configuration).  Results are identical for every choice."""
    _check(_lib_or_raise().qstate_set_scan_partitions(int(n)))


def qstate_scan_partition_count(cfg: Config, x: Inputs, stats: Stats) -> int:
    """Batch partitions a scan with these arguments would use now (0 if they are invalid)."""
    c, xi, st = cfg.c(), x.c(), stats.c()
    return int(_lib_or_raise().qstate_scan_partition_count(ct.byref(c), ct.byref(xi), ct.byref(st)))
