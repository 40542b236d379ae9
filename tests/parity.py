"""Helpers of the GPU parity tests: host <-> device copies of states and the comparisons of
the lockstep protocol.  Data flows one way: oracle states and inputs are given to the GPU,
and GPU results are checked against the oracle's -- never fed back into it."""
from __future__ import annotations

import numpy as np

REL_O_QUANT = 1e-3     # readout tolerance of the quantised path, max relative per vector
REL_O_LOCKSTEP = 1e-5  # readouts of a write-back started from the oracle's own packed state,
                       # normwise over the heads of a token: both sides dequantise the same codes
                       # and read out before quantising (Sec. 2), so they differ by FP32 rounding
                       # only.  Per vector the relative error also measures the conditioning of
                       # S^T q: where the state's columns nearly cancel against q (at a first
                       # write-back from the zero state o = u (k . q), and k . q can be ~1e-3)
                       # any change of summation order moves it by far more than 1e-5.
REL_O_FP32 = 1e-5      # readout tolerance of the unquantised FP32 path
REL_STATS = 1e-5       # EMA statistics and row ranges
CODE_AGREE = 0.9999    # fraction of identical state codes
NEAR_TIE = 1e-5        # relative SSE gap under which two fitted factors are both correct
WIDE_BITS = 8          # CODE_AGREE applies to rows up to this width; wider rows: per code


def near_boundary(x, D, R, rel=REL_STATS):
    """For a wider row the identical-code bar is finer than FP32 can settle: at b bits a step is
    about R / 2^(b-1), so state values that agree within rel * R (the tolerance of the row
    ranges) round to different codes wherever the exact value lies within rel * R of a rounding
    boundary.  True where x / D lies within rel * R / D of a half-integer, in the oracle's
    operations (FP32 x * (1 / D))."""
    x = np.asarray(x, np.float32)
    D = np.asarray(D, np.float32)
    inv = np.where(D > 0, np.float32(1.0) / np.where(D > 0, D, np.float32(1.0)), np.float32(0.0))
    u = np.abs((x * inv).astype(np.float32)).astype(np.float64)
    dist = np.abs(u - (np.floor(u) + 0.5))
    return dist <= rel * np.asarray(R, np.float64) * inv.astype(np.float64) + 1e-12


def dev(a, torch, device="cuda"):
    a = np.ascontiguousarray(a)
    if a.dtype == np.uint16:
        a = a.view(np.int16)
    elif a.dtype == np.uint32:
        a = a.view(np.int32)
    return torch.from_numpy(a.copy()).to(device)


def host(t, dtype):
    a = t.detach().cpu().numpy()
    return a.view(dtype) if a.dtype.itemsize == np.dtype(dtype).itemsize else a.astype(dtype)


def to_gpu_state(q, torch, cfg, buf):
    return q.State(dev(buf.payload, torch), dev(buf.scales, torch), dev(buf.widths, torch),
                   dev(buf.head_off, torch), dev(buf.fidx, torch))


def set_gpu_state(st, buf, b=None, region=None, units=None, groups=None, H=None):
    """Copy an oracle Buf into GPU State tensors (whole, or batch element b only)."""
    import torch
    def put(t, a, lo=None, hi=None):
        src = torch.from_numpy(np.ascontiguousarray(a).view(
            {np.dtype(np.uint16): np.int16, np.dtype(np.uint32): np.int32}.get(a.dtype, a.dtype)))
        if lo is None:
            t.copy_(src.to(t.device))
        else:
            t[lo:hi].copy_(src.to(t.device))
    if b is None:
        for t, a in zip((st.payload, st.scales, st.widths, st.head_off, st.fidx),
                        (buf.payload, buf.scales, buf.widths, buf.head_off, buf.fidx)):
            put(t, a)
    else:
        put(st.payload, buf.payload, b * region, (b + 1) * region)
        put(st.scales, buf.scales, b * groups, (b + 1) * groups)
        put(st.fidx, buf.fidx, b * groups, (b + 1) * groups)
        put(st.widths, buf.widths, b * units, (b + 1) * units)
        put(st.head_off, buf.head_off, b * H, (b + 1) * H)


def from_gpu_state(orc, st):
    return orc.Buf(host(st.payload, np.uint8), host(st.scales, np.uint16), host(st.widths, np.uint8),
                   host(st.head_off, np.uint32), host(st.fidx, np.uint8))


def rel_err_vectors(a, ref):
    """max over vectors (last axis) of |a - ref| / max(|ref|, 1e-30)."""
    a = a.astype(np.float64)
    ref = ref.astype(np.float64)
    num = np.linalg.norm(a - ref, axis=-1)
    den = np.maximum(np.linalg.norm(ref, axis=-1), 1e-30)
    return float(np.max(num / den)) if num.size else 0.0


def rel_err_tokens(a, ref):
    """Readouts (B, T, H, dv): max over tokens t of the normwise relative error of all of token
    t's readouts, |a[:, t] - ref[:, t]|_F / max(|ref[:, t]|_F, 1e-30)."""
    a = np.asarray(a, np.float64)
    ref = np.asarray(ref, np.float64)
    if ref.size == 0:
        return 0.0
    num = np.sqrt(np.sum((a - ref) ** 2, axis=(0, 2, 3)))
    den = np.maximum(np.sqrt(np.sum(ref ** 2, axis=(0, 2, 3))), 1e-30)
    return float(np.max(num / den))


def cand_step(k, R, b):
    """Candidate step k of a group of range R at width b >= 2 (reading R3 of Sec. 3's fit):
    FP16(fl(fl(f_k R) fl(1/n))), saturated at 65504, as float32."""
    n = 2 ** (b - 1) - 1
    f = np.float32(5 + k) / np.float32(20)
    v = np.float32(np.float32(f * np.float32(R)) * (np.float32(1.0) / np.float32(n)))
    return np.float32(np.float16(min(v, np.float32(65504.0))))


def range_samples(R, b, rel=REL_STATS):
    """Ranges R' within rel * R of R, one inside each sub-interval on which every candidate
    step FP16(f_k R' / n) is constant (the steps change only where f_k R' / n crosses an FP16
    rounding boundary): the ranges that a computation agreeing with R within rel may have seen."""
    lo = np.float32(np.float64(R) * (1.0 - rel))
    hi = np.float32(np.float64(R) * (1.0 + rel))
    pts = {lo, hi, np.float32(R)}
    for k in range(16):
        if cand_step(k, lo, b) == cand_step(k, hi, b):
            continue
        a, z = lo, hi                     # bisect for the first R' with the upper step
        target = cand_step(k, hi, b)
        while np.nextafter(a, np.float32(np.inf)) < z:
            m = np.float32((np.float64(a) + np.float64(z)) / 2)
            if m <= a or m >= z:
                break
            if cand_step(k, m, b) == target:
                z = m
            else:
                a = m
        pts.update((a, z))
    return sorted(pts)


def factor_explained_by_range(x, b, fid, D, R_ref, R_gpu=None):
    """True if fitted factor fid with stored step D is the argmin (within NEAR_TIE) of the
    squared errors of the group x under the candidate steps built from a range the GPU may have
    seen: its own stored range R_gpu (row unit), else any range within REL_STATS of the
    oracle's R_ref; the step of fid under that range must be D (Sec. 3, R23 of the readings)."""
    rs = [np.float32(R_gpu)] if R_gpu is not None else range_samples(R_ref, b)
    for r in rs:
        if cand_step(fid, r, b) != np.float32(D):
            continue
        sse = candidate_sse(x, b, r)
        if sse[fid] <= sse.min() * (1 + NEAR_TIE) + 1e-30:
            return True
    return False


def codes_of(orc, cfg, buf):
    """Codes (B, H, dk, dv) and widths (B, H, dk) of a packed state, decoded row by row by the
    oracle's layout function (slow; the reference for :func:`codes_fast`)."""
    B, H, dk, dv = cfg.B, cfg.H, cfg.dk, cfg.dv
    rb = cfg.region_bytes
    w = buf.widths.reshape(B, -1)
    if cfg.unit_kind == 1:
        w = np.repeat(w, dk, axis=1)
    w = w.reshape(B, H, dk).astype(int)
    out = np.zeros((B, H, dk, dv), np.int64)
    for b in range(B):
        for h in range(H):
            off = b * rb + int(buf.head_off[b * H + h])
            for i in range(dk):
                nb = w[b, h, i] * dv // 8
                if nb:
                    out[b, h, i] = orc.unpack_codes(buf.payload[off:off + nb], dv, w[b, h, i])
                off += nb
    return out, w


def codes_fast(cfg, buf):
    """Codes (B, H, dk, dv) and widths (B, H, dk) of a packed state, all rows of one width at a
    time: row element j's code is row bits [j w, j w + w), bit m of a row being bit m % 8 of
    byte m / 8 (the storage layout of Sec. 3 as this library reads it).  Pinned against the
    oracle's row decoder on the CPU."""
    B, H, dk, dv = cfg.B, cfg.H, cfg.dk, cfg.dv
    rb = cfg.region_bytes
    w = buf.widths.reshape(B, -1).astype(np.int64)
    if cfg.unit_kind == 1:
        w = np.repeat(w, dk, axis=1)
    w = w.reshape(B, H, dk)
    row_bytes = w * (dv // 8)
    start = (np.arange(B, dtype=np.int64)[:, None, None] * rb
             + buf.head_off.reshape(B, H, 1).astype(np.int64)
             + np.cumsum(row_bytes, axis=2) - row_bytes)
    out = np.zeros((B, H, dk, dv), np.int64)
    wf, sf, of = w.reshape(-1), start.reshape(-1), out.reshape(-1, dv)
    for b in np.unique(wf):
        if b == 0:
            continue
        rows = np.nonzero(wf == b)[0]
        nb = int(b) * dv // 8
        by = buf.payload[sf[rows][:, None] + np.arange(nb)]
        bits = np.unpackbits(by, axis=1, bitorder="little").reshape(rows.size, dv, int(b))
        of[rows] = (bits.astype(np.int64) << np.arange(int(b))).sum(axis=2)
    return out, w.astype(int)


def candidate_sse(x, b, R):
    """Squared errors (FP64) of the 16 candidate steps of a group x at width b >= 2 when the
    steps are built from the range R (reading R3 of Sec. 3's fit: Delta_k =
    FP16(fl(fl(f_k R) fl(1/n))), q = clamp(rint(fl(x / Delta)), -n, n))."""
    x = np.asarray(x, np.float32)
    n = 2 ** (b - 1) - 1
    R = np.float32(R)
    inv_n = np.float32(1.0) / np.float32(n)
    out = np.zeros(16)
    for k in range(16):
        f = np.float32(5 + k) / np.float32(20)
        D = np.float32(np.float16(np.float32(np.float32(f * R) * inv_n)))
        inv = np.float32(0.0) if D == 0 else np.float32(1.0) / D
        q = np.clip(np.rint((x * inv).astype(np.float32)), -n, n)
        e = x.astype(np.float64) - q.astype(np.float64) * np.float64(D)
        out[k] = float(np.sum(e * e))
    return out


def compare_packed(orc, cfg, gpu: "orc.Buf", ref: "orc.Buf", X=None, max_tie_frac=5e-4, R_gpu=None,
                   R_ref=None):
    """Compare a GPU-written packed state with the oracle's for the same target widths.

    Widths/offsets must be equal.  Fitted factors may differ only where the oracle's own
    candidate errors (FP64, from its pre-quantisation state X) tie within NEAR_TIE, or (row
    unit, given the GPU's row ranges R_gpu, which agree with the oracle's R_ref within
    REL_STATS) where the GPU's factor is the argmin of the oracle state's errors under the
    candidate steps built from R_gpu: a step FP16(f R / n) that lies within R's last-ulp
    differences of an FP16 rounding boundary rounds to the neighbouring FP16 number, which
    changes that candidate's error.  Such groups are rare and are checked by these criteria
    instead of code equality.  Elsewhere at least CODE_AGREE of the codes are identical and
    the rest differ by one step; scales are identical up to a rare one-ulp FP16 difference
    traced to last-ulp differences of R."""
    assert np.array_equal(gpu.widths, ref.widths)
    assert np.array_equal(gpu.head_off, ref.head_off)
    cg, w = codes_fast(cfg, gpu)
    cr, _ = codes_fast(cfg, ref)
    B, H, dk, dv = cfg.B, cfg.H, cfg.dk, cfg.dv
    fid_g, fid_r = gpu.fidx.astype(int), ref.fidx.astype(int)
    sc_g, sc_r = gpu.scales.astype(np.int64), ref.scales.astype(np.int64)
    # scale-group mask per element
    if cfg.unit_kind == 0:
        gmask_of = lambda m: np.broadcast_to(m.reshape(B, H, dk, 1), (B, H, dk, dv))
    else:
        gmask_of = lambda m: np.repeat(m.reshape(B, H, dk // 32, 1, dv), 32, axis=3).reshape(B, H, dk, dv)
    diff_fid = fid_g != fid_r
    wflat = (w.reshape(-1) if cfg.unit_kind == 0 else
             np.repeat(w[:, :, ::32][..., None], dv, axis=-1).reshape(-1))
    diff_fid &= wflat >= 2     # factors of width 0/1 groups are carried, not fitted
    ties = int(diff_fid.sum())
    stats = dict(groups=int(fid_g.size), fidx_diff=ties)
    if ties:
        assert X is not None, "fitted factors differ and no oracle state to check ties"
        assert ties <= max(2, max_tie_frac * fid_g.size), stats
        idx = np.nonzero(diff_fid)[0]
        for gidx in idx:
            xs = _group_values(cfg, X, gidx)
            b = int(wflat[gidx])
            _, _, _, sse = orc.quant_group(xs, b, with_sse=True)
            m = sse.min()
            if sse[fid_g[gidx]] <= m * (1 + NEAR_TIE) + 1e-30:
                continue
            # the GPU's range builds a different FP16 step for some candidate (R23)
            rr = float(np.max(np.abs(xs)))
            rg = None
            if R_gpu is not None and cfg.unit_kind == 0:
                rg = float(R_gpu[gidx])
                assert abs(rg - rr) <= REL_STATS * rr, (gidx, rg, rr)
            Dg = np.float32(gpu.scales[gidx:gidx + 1].view(np.float16)[0])
            assert factor_explained_by_range(xs, b, int(fid_g[gidx]), Dg, rr, rg), \
                (gidx, sse, fid_g[gidx], fid_r[gidx])
    same = ~gmask_of(diff_fid)
    dd = np.abs(cg - cr)
    wel = np.broadcast_to(w[..., None], cg.shape)
    narrow, wide = same & (wel <= WIDE_BITS), same & (wel > WIDE_BITS)
    d = dd[narrow]
    agree = float(np.mean(d == 0)) if d.size else 1.0
    stats.update(code_agree=agree, code_maxdiff=int(d.max()) if d.size else 0)
    assert agree >= CODE_AGREE, stats
    assert (d.max() if d.size else 0) <= 1, stats
    if wide.any():
        # wider rows: the GPU's codes against the oracle's state quantised with the GPU's own
        # stored step (a one-ulp FP16 step difference, allowed below, moves a code at |x| near
        # R by about n 2^-10 steps, i.e. several at 12 bits and more); each differs by at most
        # one step, and only at a value within the range tolerance of a rounding boundary
        assert X is not None, "wide rows need the oracle state"
        Xe = np.asarray(X, np.float32).reshape(cg.shape)
        Dg = gpu.scales.view(np.float16).astype(np.float32)
        if cfg.unit_kind == 0:
            Dg = np.broadcast_to(Dg.reshape(B, H, dk, 1), cg.shape)
            Rg = np.broadcast_to(np.abs(Xe).max(axis=-1, keepdims=True), cg.shape)
        else:
            Dg = np.repeat(Dg.reshape(B, H, dk // 32, 1, dv), 32, axis=3).reshape(cg.shape)
            Rb = np.abs(Xe).reshape(B, H, dk // 32, 32, dv).max(axis=3, keepdims=True)
            Rg = np.repeat(Rb, 32, axis=3).reshape(cg.shape)
        xw, Dw, Rw = Xe[wide], Dg[wide], Rg[wide]
        nw = (2 ** (wel[wide] - 1) - 1).astype(np.float64)
        inv = np.where(Dw > 0, np.float32(1.0) / np.where(Dw > 0, Dw, np.float32(1.0)), np.float32(0.0))
        q_exp = np.clip(np.rint((xw * inv).astype(np.float32)).astype(np.float64), -nw, nw)
        dq = np.abs((cg[wide] - nw) - q_exp)
        flip = dq != 0
        stats.update(wide_code_agree=float(1.0 - flip.mean()), wide_maxdiff=int(dq.max()))
        assert dq.max() <= 1, stats
        ok = near_boundary(xw[flip], Dw[flip], Rw[flip])
        assert ok.all(), (stats, int((~ok).sum()))
    # scales: equal where factors agree, up to rare one-ulp FP16 differences, each of which must
    # be the step of the group's factor under a range the GPU may have seen (its own stored
    # range for the row unit, else one within REL_STATS of the oracle's): ranges that agree
    # within FP32 rounding straddle an FP16 rounding boundary of f R / n now and then
    sd_all = np.abs(sc_g - sc_r)
    sd = sd_all[~diff_fid]
    stats.update(scale_diff=int(np.sum(sd != 0)))
    assert np.all(sd <= 1), stats
    assert np.sum(sd != 0) <= max(2, 1e-2 * sd.size), stats
    for gidx in np.nonzero((sd_all != 0) & ~diff_fid)[0]:
        assert X is not None, "scales differ and no oracle state to check them"
        xs = np.asarray(_group_values(cfg, X, gidx), np.float32)
        b = int(wflat[gidx])
        Dg = np.float32(gpu.scales[gidx:gidx + 1].view(np.float16)[0])
        if b >= 2:
            rr = np.float32(np.max(np.abs(xs)))
            if R_gpu is not None and cfg.unit_kind == 0:
                ok = cand_step(int(fid_g[gidx]), np.float32(R_gpu[gidx]), b) == Dg
            else:
                lo, hi = (cand_step(int(fid_g[gidx]), r, b) for r in (range_samples(rr, b)[0], range_samples(rr, b)[-1]))
                ok = lo <= Dg <= hi
        else:   # one bit: FP16 of the mean magnitude
            m = np.float64(np.sum(np.abs(xs), dtype=np.float64)) / xs.size
            lo, hi = (np.float32(np.float16(np.float32(m * f))) for f in (1 - REL_STATS, 1 + REL_STATS))
            ok = lo <= Dg <= hi
        assert ok, (stats, int(gidx), b, float(Dg))
    return stats


def _group_values(cfg, X, gidx):
    B, H, dk, dv = cfg.B, cfg.H, cfg.dk, cfg.dv
    if cfg.unit_kind == 0:
        return X.reshape(-1, dv)[gidx]
    nb = dk // 32
    bh, rem = divmod(gidx, nb * dv)
    blk, j = divmod(rem, dv)
    return X.reshape(B * H, dk, dv)[bh, blk * 32:(blk + 1) * 32, j]
