"""ctypes wrapper of ``qstate_oracle.c`` (plain CPU reference; test infrastructure only).

Arrays are numpy, host memory, C-contiguous.  Layouts are the library's:

* state payload: ``B`` regions of ``region_bytes`` bytes; head ``h`` of batch element ``b`` at
  byte ``head_off[b*H + h]`` inside its region, rows in order, row ``i`` ``width*dv/8`` bytes;
* scales (FP16 bits, uint16) and fitted-factor indices (uint8): one per scale group --
  ``(B, H, dk)`` for the row unit, ``(B, H, dk/32, dv)`` for the head unit;
* widths (uint8): ``(B, H, dk)`` row unit, ``(B, H)`` head unit; statistics ``ema_s, ema_r,
  range`` (float32) per unit.
"""
from __future__ import annotations

import ctypes as ct
import os
import subprocess
from dataclasses import dataclass

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "qstate_oracle.c")
_LIB = os.path.join(_HERE, "_build", "liborc.so")
# timing build: the same source with a write-back's heads shared out over OpenMP threads
# (identical arithmetic per head); the checker is always the plain single-thread build
_LIB_OMP = os.path.join(_HERE, "_build", "liborc_omp.so")
_FLAGS = ["-std=c11", "-O2", "-ffp-contract=off", "-fno-fast-math", "-fPIC", "-shared"]


def _gcc(out, extra):
    if not os.path.exists(out) or os.path.getmtime(out) < os.path.getmtime(_SRC):
        os.makedirs(os.path.dirname(out), exist_ok=True)
        tmp = out + f".{os.getpid()}.tmp"
        subprocess.check_call(["gcc", *_FLAGS, *extra, "-o", tmp, _SRC, "-lm"])
        os.replace(tmp, out)
    return out


def build(force: bool = False) -> str:
    """Compile the oracle with gcc (no FMA contraction, no fast-math)."""
    if force and os.path.exists(_LIB):
        os.remove(_LIB)
    return _gcc(_LIB, [])


def build_parallel() -> str:
    """Compile the OpenMP timing build (heads of a write-back in parallel; used only to time
    the oracle on all host cores)."""
    return _gcc(_LIB_OMP, ["-fopenmp", "-DORC_OPENMP"])


class OrcCfg(ct.Structure):
    _fields_ = [("B", ct.c_int32), ("H", ct.c_int32), ("dk", ct.c_int32), ("dv", ct.c_int32),
                ("decay_kind", ct.c_int32), ("erase_kind", ct.c_int32),
                ("unit_kind", ct.c_int32), ("group_heads", ct.c_int32),
                ("bbar_num", ct.c_int32), ("bbar_den", ct.c_int32), ("bmin", ct.c_int32),
                ("bmax", ct.c_int32), ("C", ct.c_int32), ("fit_every", ct.c_int32),
                ("ema_span", ct.c_float), ("gate_bits", ct.c_int32),
                ("weight_kind", ct.c_int32), ("alloc_mode", ct.c_int32)]


@dataclass
class Cfg:
    """Method configuration (mirrors the library's; kept separate on purpose)."""
    B: int
    H: int
    dk: int
    dv: int
    decay_kind: int = 0      # 0 per row, 1 per head
    erase_kind: int = 0      # 0 delta rule, 1 none, 2 general (a, w given per token)
    unit_kind: int = 0       # 0 row unit, 1 head unit
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
    alloc_mode: int = 0      # 0 lagged widths, 1 widths from this write-back's statistics

    def c(self) -> OrcCfg:
        return OrcCfg(*[getattr(self, f) for f, _ in OrcCfg._fields_])

    @property
    def units(self) -> int:
        return self.H * self.dk if self.unit_kind == 0 else self.H

    @property
    def n_scale_groups(self) -> int:
        return self.H * self.dk if self.unit_kind == 0 else self.H * (self.dk // 32) * self.dv

    @property
    def region_bytes(self) -> int:
        return self.H * self.dk * self.dv * self.bbar_num // (8 * self.bbar_den)

    @classmethod
    def from_workload(cls, w, **over) -> "Cfg":
        kw = dict(B=w.B, H=w.H, dk=w.dk, dv=w.dv, decay_kind=0 if w.per_row_decay else 1,
                  erase_kind=(2 if getattr(w, "general", False) else 0 if w.erase else 1),
                  unit_kind=0 if w.unit == "row" else 1,
                  group_heads=w.group_heads, bbar_num=w.bbar, bbar_den=1, bmin=w.bmin,
                  bmax=w.bmax, C=w.C, gate_bits=w.gate_bits)
        kw.update(over)
        return cls(**kw)


_lib = None
_lib_par = None


def lib(parallel: bool = False):
    """The plain build (the checker), or with ``parallel`` the OpenMP timing build."""
    global _lib, _lib_par
    if parallel:
        if _lib_par is None:
            _lib_par = _declare(ct.CDLL(build_parallel()))
        return _lib_par
    if _lib is None:
        _lib = _declare(ct.CDLL(build()))
    return _lib


def _declare(L):
    """Argument and result types of the exported functions."""
    P = ct.c_void_p
    L.orc_bits_per_element.restype = ct.c_double
    L.orc_bits_per_element.argtypes = [ct.POINTER(OrcCfg)]
    L.orc_expm1_series.restype = ct.c_float
    L.orc_expm1_series.argtypes = [ct.c_float]
    L.orc_recur_f32.argtypes = [ct.c_int] * 3 + [P] * 8
    L.orc_recur_f64.argtypes = [ct.c_int] * 3 + [P] * 8
    L.orc_quant_group.argtypes = [P, ct.c_int, ct.c_int, ct.c_int, ct.c_int, ct.c_int,
                                  P, P, P, P]
    L.orc_dequant_group.argtypes = [P, ct.c_int, ct.c_int, ct.c_uint16, P, ct.c_int]
    L.orc_pack_codes.argtypes = [P, ct.c_int, ct.c_int, P]
    L.orc_unpack_codes.argtypes = [P, ct.c_int, ct.c_int, P]
    L.orc_region_bytes.restype = ct.c_long
    L.orc_region_bytes.argtypes = [ct.POINTER(OrcCfg)]
    L.orc_pack.argtypes = [ct.POINTER(OrcCfg)] + [P] * 7
    L.orc_unpack.argtypes = [ct.POINTER(OrcCfg)] + [P] * 5
    L.orc_weights.argtypes = [ct.POINTER(OrcCfg), ct.c_int, P, P, P, P]
    L.orc_shuffle.argtypes = [ct.c_int, ct.POINTER(ct.c_int), ct.POINTER(ct.c_int)]
    L.orc_alloc_from_weights.argtypes = [ct.c_int, P, ct.c_int, ct.c_int, ct.c_long,
                                         ct.c_int, ct.c_int, P]
    L.orc_alloc.argtypes = [ct.POINTER(OrcCfg), P, P, P, P, P]
    L.orc_init_widths.argtypes = [ct.POINTER(OrcCfg), P, P]
    L.orc_quant_decay.argtypes = [ct.c_long, ct.c_int, P, ct.c_int, P, P, P]
    L.orc_step.argtypes = ([ct.POINTER(OrcCfg)] + [P] * 10 + [ct.c_int] * 4 + [P] * 14)
    L.orc_step_current.argtypes = ([ct.POINTER(OrcCfg)] + [P] * 10 + [ct.c_int] * 4 + [P] * 14)
    return L


def _p(a):
    return None if a is None else a.ctypes.data_as(ct.c_void_p)


def _c(a, dtype):
    a = np.ascontiguousarray(a, dtype=dtype)
    return a


def _check(rc, what):
    if rc != 0:
        raise ValueError(f"oracle {what} failed with status {rc}")


# ---------------------------------------------------------------------------------------
# Eq. (1), unquantised.
# ---------------------------------------------------------------------------------------
def recur(S0, k, q, v, s, a, w, dtype=np.float32):
    """One head, T tokens.  ``S0`` (dk, dv); ``k, q, a, s`` (T, dk); ``v, w`` (T, dv).
    Returns ``(o (T, dv), S_T)`` in ``dtype`` (float32 or float64)."""
    T, dk = k.shape
    dv = v.shape[1]
    args = [_c(x, np.float32) for x in (k, q, v, s, a, w)]
    S = np.array(S0, dtype=dtype, order="C", copy=True)
    o = np.zeros((T, dv), dtype)
    fn = lib().orc_recur_f32 if dtype == np.float32 else lib().orc_recur_f64
    fn(dk, dv, T, _p(S), *[_p(x) for x in args], _p(o))
    return o, S


def expand_inputs(cfg: Cfg, inp: dict, b: int, h: int):
    """Per-token (k, q, v, s_row, a, w) of head (b, h) for :func:`recur` (plain Eq. 1 forms:
    KDA/GDN a = beta k, w = beta 1; Mamba-2 a = 0, w = 1)."""
    k = inp["k"][b, :, h].astype(np.float32)
    q = inp["q"][b, :, h].astype(np.float32)
    v = inp["v"][b, :, h].astype(np.float32)
    T = k.shape[0]
    s = inp["s"][b, :, h]
    if s.ndim == 1:
        s = np.repeat(s[:, None], cfg.dk, axis=1)
    if cfg.erase_kind == 0:
        beta = inp["beta"][b, :, h].astype(np.float32)
        a = (beta[:, None] * k).astype(np.float32)
        w = np.repeat(beta[:, None], cfg.dv, axis=1).astype(np.float32)
    elif cfg.erase_kind == 2:
        a = inp["a"][b, :, h].astype(np.float32)
        w = inp["w"][b, :, h].astype(np.float32)
    else:
        a = np.zeros_like(k)
        w = np.ones((T, cfg.dv), np.float32)
    return k, q, v, s.astype(np.float32), a, w


# ---------------------------------------------------------------------------------------
# Levels and storage.
# ---------------------------------------------------------------------------------------
def quant_group(x, b, refit=True, fidx_in=15, with_sse=False):
    x = _c(x, np.float32)
    g = x.size
    codes = np.zeros(g, np.uint16)
    scale = np.zeros(1, np.uint16)
    fidx = np.zeros(1, np.uint8)
    sse = np.zeros(16, np.float64)
    lib().orc_quant_group(_p(x), g, 1, b, int(refit), int(fidx_in), _p(codes), _p(scale),
                          _p(fidx), _p(sse))
    out = (codes, int(scale[0]), int(fidx[0]))
    return out + (sse,) if with_sse else out


def dequant_group(codes, b, scale):
    codes = _c(codes, np.uint16)
    x = np.zeros(codes.size, np.float32)
    lib().orc_dequant_group(_p(codes), codes.size, b, int(scale), _p(x), 1)
    return x


def pack_codes(codes, b):
    codes = _c(codes, np.uint16)
    dst = np.zeros(b * codes.size // 8, np.uint8)
    lib().orc_pack_codes(_p(codes), codes.size, b, _p(dst))
    return dst


def unpack_codes(src, g, b):
    src = _c(src, np.uint8)
    codes = np.zeros(g, np.uint16)
    lib().orc_unpack_codes(_p(src), g, b, _p(codes))
    return codes


def bits_per_element(cfg: Cfg) -> float:
    c = cfg.c()
    return lib().orc_bits_per_element(ct.byref(c))


def init_widths(cfg: Cfg):
    widths = np.zeros(cfg.B * cfg.units, np.uint8)
    head_off = np.zeros(cfg.B * cfg.H, np.uint32)
    c = cfg.c()
    _check(lib().orc_init_widths(ct.byref(c), _p(widths), _p(head_off)), "init_widths")
    return widths, head_off


def pack(cfg: Cfg, S, widths, head_off):
    """Quantise + pack a dense state ``S`` (B, H, dk, dv); returns payload, scales, fidx, range."""
    S = _c(S, np.float32)
    widths = _c(widths, np.uint8)
    head_off = _c(head_off, np.uint32)
    payload = np.zeros(cfg.B * cfg.region_bytes, np.uint8)
    scales = np.zeros(cfg.B * cfg.n_scale_groups, np.uint16)
    fidx = np.zeros(cfg.B * cfg.n_scale_groups, np.uint8)
    rng = np.zeros(cfg.B * cfg.units, np.float32)
    c = cfg.c()
    _check(lib().orc_pack(ct.byref(c), _p(S), _p(widths), _p(head_off), _p(payload), _p(scales),
                          _p(fidx), _p(rng)), "pack")
    return payload, scales, fidx, rng


def unpack(cfg: Cfg, payload, scales, widths, head_off):
    S = np.zeros((cfg.B, cfg.H, cfg.dk, cfg.dv), np.float32)
    c = cfg.c()
    args = [_c(payload, np.uint8), _c(scales, np.uint16), _c(widths, np.uint8),
            _c(head_off, np.uint32)]
    _check(lib().orc_unpack(ct.byref(c), *[_p(a) for a in args], _p(S)), "unpack")
    return S


# ---------------------------------------------------------------------------------------
# Allocation (Eq. 3, Eq. 4 + rounding).
# ---------------------------------------------------------------------------------------
def weights(cfg: Cfg, ema_s, ema_r, rng, b=0):
    """FP32 weights c of batch element b; the null weight (below 2^-60) is returned as 0."""
    c = cfg.c()
    out = np.zeros(cfg.units, np.float32)
    args = [_c(ema_s, np.float32), _c(ema_r, np.float32), _c(rng, np.float32)]
    _check(lib().orc_weights(ct.byref(c), b, *[_p(a) for a in args], _p(out)), "weights")
    return np.where(out < 0, 0.0, out).astype(np.float32)


def shuffle_map(N):
    """The shuffled-decay bijection of N units (weight kind 7): u -> (A u + B) mod N."""
    A, B = ct.c_int(), ct.c_int()
    lib().orc_shuffle(N, ct.byref(A), ct.byref(B))
    return (A.value * np.arange(N, dtype=np.int64) + B.value) % N


def alloc_from_weights(cw, bmin, bmax, total, bbar_num=None, bbar_den=1):
    """Integer widths for weights ``cw`` (float32; 0 = null weight) summing to ``total``."""
    cw = np.where(np.asarray(cw, np.float32) > 0, cw, -1.0).astype(np.float32)
    N = cw.size
    if bbar_num is None:
        bbar_num, bbar_den = total, N
    widths = np.zeros(N, np.uint8)
    rc = lib().orc_alloc_from_weights(N, _p(cw), bmin, bmax, total, bbar_num, bbar_den,
                                      _p(widths))
    if rc == 2:
        raise ValueError("infeasible budget")
    _check(rc, "alloc_from_weights")
    return widths


def alloc(cfg: Cfg, ema_s, ema_r, rng):
    widths = np.zeros(cfg.B * cfg.units, np.uint8)
    head_off = np.zeros(cfg.B * cfg.H, np.uint32)
    c = cfg.c()
    args = [_c(ema_s, np.float32), _c(ema_r, np.float32), _c(rng, np.float32)]
    rc = lib().orc_alloc(ct.byref(c), *[_p(a) for a in args], _p(widths), _p(head_off))
    if rc == 2:
        raise ValueError("infeasible budget")
    _check(rc, "alloc")
    return widths, head_off


def expm1_series(x: float) -> float:
    return float(lib().orc_expm1_series(float(x)))


# ---------------------------------------------------------------------------------------
# Log-uniform decay-gate quantiser.
# ---------------------------------------------------------------------------------------
def quant_decay(s, nchan, g):
    """``s`` (..., nchan) float32 > 0 -> codes (same shape, uint8), LUT (nchan, 2^g),
    thresholds (nchan, 2^g - 1)."""
    s = _c(s, np.float32)
    count = s.size // nchan
    L = 1 << g
    codes = np.zeros(s.shape, np.uint8)
    lut = np.zeros((nchan, L), np.float32)
    thr = np.zeros((nchan, L - 1), np.float32)
    _check(lib().orc_quant_decay(count, nchan, _p(s), g, _p(codes), _p(lut), _p(thr)),
           "quant_decay")
    return codes, lut, thr


# ---------------------------------------------------------------------------------------
# One write-back interval for all heads.
# ---------------------------------------------------------------------------------------
@dataclass
class Buf:
    payload: np.ndarray
    scales: np.ndarray
    widths: np.ndarray
    head_off: np.ndarray
    fidx: np.ndarray

    def copy(self) -> "Buf":
        return Buf(*(a.copy() for a in (self.payload, self.scales, self.widths, self.head_off,
                                          self.fidx)))


def new_buf(cfg: Cfg) -> Buf:
    return Buf(np.zeros(cfg.B * cfg.region_bytes, np.uint8),
               np.zeros(cfg.B * cfg.n_scale_groups, np.uint16),
               np.zeros(cfg.B * cfg.units, np.uint8), np.zeros(cfg.B * cfg.H, np.uint32),
               np.full(cfg.B * cfg.n_scale_groups, 15, np.uint8))


def init_state(cfg: Cfg):
    """Zero state packed with the initial (uniform) widths, in both buffers."""
    widths, head_off = init_widths(cfg)
    S0 = np.zeros((cfg.B, cfg.H, cfg.dk, cfg.dv), np.float32)
    payload, scales, fidx, _ = pack(cfg, S0, widths, head_off)
    a = Buf(payload, scales, widths.copy(), head_off.copy(), fidx)
    b = new_buf(cfg)
    b.widths[:] = widths
    b.head_off[:] = head_off
    return a, b


def step(cfg: Cfg, src: Buf, dst: Buf, inp: dict, t_begin, t_end, w_index, o, ema_s, ema_r,
         rng, s_code=None, s_lut=None, want_x=False, parallel=False):
    """Run tokens [t_begin, t_end) from ``src`` into ``dst`` (whose widths/offsets are the
    target).  ``inp`` holds the full (B, T, H, .) inputs; ``o`` (B, T, H, dv) is written.
    Returns the FP32 pre-quantisation state if ``want_x``.  ``parallel`` runs the OpenMP
    timing build (same results)."""
    T = inp["q"].shape[1]
    c = cfg.c()
    x = np.zeros((cfg.B, cfg.H, cfg.dk, cfg.dv), np.float32) if want_x else None
    q, k, v = (_c(inp[n], np.float32) for n in ("q", "k", "v"))
    s = None if s_code is not None else _c(inp["s"], np.float32)
    beta = _c(inp["beta"], np.float32)
    a_in = _c(inp["a"], np.float32) if "a" in inp else None
    w_in = _c(inp["w"], np.float32) if "w" in inp else None
    sc = None if s_code is None else _c(s_code, np.uint8)
    sl = None if s_lut is None else _c(s_lut, np.float32)
    fn = lib().orc_step_current if cfg.alloc_mode == 1 else lib(parallel).orc_step
    rc = fn(ct.byref(c), _p(src.payload), _p(src.scales), _p(src.widths),
                        _p(src.head_off), _p(src.fidx), _p(dst.payload), _p(dst.scales),
                        _p(dst.widths), _p(dst.head_off), _p(dst.fidx), T, t_begin, t_end,
                        w_index, _p(q), _p(k), _p(v), _p(s), _p(sc), _p(sl), _p(beta), _p(o),
                        _p(ema_s), _p(ema_r), _p(rng), _p(x), _p(a_in), _p(w_in))
    _check(rc, "step")
    return x


def scan(cfg: Cfg, inp: dict, T=None, s_code=None, s_lut=None):
    """Free-running quantised scan from the zero state.  Returns (o, final Buf, ema_s, ema_r,
    range)."""
    T = inp["q"].shape[1] if T is None else T
    src, dst = init_state(cfg)
    o = np.zeros((cfg.B, inp["q"].shape[1], cfg.H, cfg.dv), np.float32)
    ema_s = np.zeros(cfg.B * cfg.units, np.float32)
    ema_r = np.zeros(cfg.B * cfg.units, np.float32)
    rng = np.zeros(cfg.B * cfg.units, np.float32)
    w = 0
    for t0 in range(0, T, cfg.C):
        t1 = min(T, t0 + cfg.C)
        step(cfg, src, dst, inp, t0, t1, w, o, ema_s, ema_r, rng, s_code, s_lut)
        if cfg.alloc_mode == 0:   # lagged: the next write-back packs with widths from these statistics
            src.widths[:], src.head_off[:] = alloc(cfg, ema_s, ema_r, rng)
        src, dst = dst, src
        w += 1
    return o, src, ema_s, ema_r, rng
