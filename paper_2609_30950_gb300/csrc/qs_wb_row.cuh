// qs_wb_row.cuh -- persistent write-back kernel for the row allocation unit (sm_103a).
//
// The hot path of qstate_step / qstate_scan for per-row widths (KDA, Mamba-2): one write-back
// interval of every head, packed state in, packed state out.
//
// Each CTA (NW warps, one CTA per SM) walks heads g = blockIdx.x, blockIdx.x + gridDim.x, ...
// While it works on head g, cp.async copies head g + gridDim.x's inputs into the other half of
// a double buffer: widths in/out, FP16 scales, fitted-factor indices, EMA statistics, the first
// token's k, q, v and rates, and the head's packed rows (whose byte window comes from offsets
// fetched one head earlier).  Warp w owns key rows [w RPW, (w+1) RPW), lane l the value
// columns [l CPL, (l+1) CPL).  Per head there are five CTA barriers:
//   B1  the head's inputs have landed            -> issue the next head's copies
//   B2  prep: row offsets (prefix sums of widths), layout checks, per-row decay, EMA update,
//       dequantisation constants with the first token's decay folded in, erase vector, k.q
//       -> unpack + dequantise into registers (column pairs), Eq. (1) partial p = a^T S',
//       r = q^T S' per lane over the warp's rows
//   B3  partials of all warps                     -> u = beta v - p, o = r + u (k.q)
//   B4  u                                         -> S = S' + k u^T; then, warp-locally:
//       row ranges, per-row steps (lane r <-> row r) or the 16 candidate steps of every row
//       (4 (row, candidate) pairs per lane), the squared-error search (candidates outer,
//       rows inner, packed FP32), codes folded into 64-bit chunks, and each group of lanes
//       holding 8 consecutive codes writing their w bytes into the output staging rows
//   B5  all rows staged                           -> vector store of the head's region and
//       coalesced stores of scales, factor indices, ranges and EMAs.
// The next head's B1 orders the reuse of stage and staging buffers.
#pragma once

#include <algorithm>

#include "qs_common.cuh"

namespace qs {

struct WbParams {
    StepParams s;       // shared parameter block (pointers, sizes, token range)
    int nheads;         // B * H
};

template <int DK, int DV>
struct alignas(16) WbStage {
    uint8_t w_in[DK], w_out[DK], fidx[DK], scode[DK];
    uint16_t sc_in[DK];
    float ms[DK], mr[DK], k[DK], q[DK], s[DK];
    float v[DV];
    float beta, rate_h, pad0, pad1;
    int in_off, in_end, out_off, ok;              // payload window of this head
    int nxt_in_off, nxt_in_end, nxt_out_off, pad2;   // offsets of the following head
};

template <int DK, int DV, int NW>
struct alignas(16) WbSmem {
    static constexpr int RPW = DK / NW;
    WbStage<DK, DV> st[2];
    float cand[DK][kNFit][2];             // (Delta_k, 1/Delta_k) per row and candidate
    uint2 chunk[NW][RPW][32];             // each lane's codes per row
    float red[2][NW][DV];                 // p and r partials per warp
    float4 deq[DK];                       // (-A, S, B, 0): x = (2^23 + u - A) S + B
    float4 wc[17];                        // per width: (n, 1/n, 2^23*1.5 - n, 2^23*1.5 + n)
    float tk[DK], tq[DK], tv[DV];         // inputs of tokens after the first (C > 1)
    float a[DK], d[DK];                   // erase vector beta k, decay of the current token
    float u[DV];
    float rowR[DK], rowM[DK];
    float fitf[kNFit];
    float wsum[NW];
    int best_k[DK];
    int off_in[DK + 1], off_out[DK + 1];
    uint16_t out_scale[DK];
    uint8_t out_fidx[DK];
    int flag;
};

// Sum N per-lane values over the warp by recursive halving; lane l ends with the total of
// value index (l >> (5 - log2 N)) & (N - 1).
template <int N>
__device__ __forceinline__ float reduce_rows(float (&v)[N], int lane) {
    constexpr int LOG = N == 16 ? 4 : N == 8 ? 3 : N == 4 ? 2 : N == 2 ? 1 : 0;
#pragma unroll
    for (int st = 0; st < LOG; ++st) {
        const int half = (N / 2) >> st;
        const int off = 16 >> st;
        const bool upper = (lane & off) != 0;
#pragma unroll
        for (int i = 0; i < half; ++i) {
            const float send = upper ? v[i] : v[i + half];
            const float keep = upper ? v[i + half] : v[i];
            v[i] = keep + __shfl_xor_sync(kFull, send, off);
        }
    }
    float t = v[0];
#pragma unroll
    for (int off = 16 >> LOG; off > 0; off >>= 1) t += __shfl_xor_sync(kFull, t, off);
    return t;
}

__device__ __forceinline__ void cp_async16(void* smem, const void* gmem) {
    const unsigned s = static_cast<unsigned>(__cvta_generic_to_shared(smem));
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;\n" ::"r"(s), "l"(gmem) : "memory");
}
__device__ __forceinline__ void cp_async8(void* smem, const void* gmem) {
    const unsigned s = static_cast<unsigned>(__cvta_generic_to_shared(smem));
    asm volatile("cp.async.ca.shared.global [%0], [%1], 8;\n" ::"r"(s), "l"(gmem) : "memory");
}
__device__ __forceinline__ void cp_async4(void* smem, const void* gmem) {
    const unsigned s = static_cast<unsigned>(__cvta_generic_to_shared(smem));
    asm volatile("cp.async.ca.shared.global [%0], [%1], 4;\n" ::"r"(s), "l"(gmem) : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;\n" ::: "memory"); }
__device__ __forceinline__ void cp_async_wait_all() { asm volatile("cp.async.wait_group 0;\n" ::: "memory"); }

// ---- packing of one row: 8 consecutive codes (w bits each) = w bytes -------------------------
// Lanes own CPL consecutive codes; groups of 8 / CPL lanes gather their chunks by shuffles and
// the group's first lane stores the w bytes at byte w * group with aligned stores.
// ALIGN16: dst is 16-byte aligned when NB == 16 (rows of dv = 128 start on 16 bytes).
template <int NB, bool ALIGN16>
__device__ __forceinline__ void store_bytes(uint8_t* dst, uint64_t lo, uint64_t hi) {
    if constexpr (NB == 16 && ALIGN16) {
        *reinterpret_cast<uint4*>(dst) = make_uint4(static_cast<uint32_t>(lo), static_cast<uint32_t>(lo >> 32),
                                                   static_cast<uint32_t>(hi), static_cast<uint32_t>(hi >> 32));
    } else if constexpr (NB == 8) {
        *reinterpret_cast<uint2*>(dst) = make_uint2(static_cast<uint32_t>(lo), static_cast<uint32_t>(lo >> 32));
    } else if constexpr (NB % 4 == 0) {
#pragma unroll
        for (int k = 0; k < NB / 4; ++k) {
            const uint64_t s = k < 2 ? lo : hi;
            reinterpret_cast<uint32_t*>(dst)[k] = static_cast<uint32_t>(s >> ((k & 1) * 32));
        }
    } else if constexpr (NB % 2 == 0) {
#pragma unroll
        for (int k = 0; k < NB / 2; ++k) {
            const uint64_t s = k < 4 ? lo : hi;
            reinterpret_cast<uint16_t*>(dst)[k] = static_cast<uint16_t>(s >> ((k & 3) * 16));
        }
    } else {
#pragma unroll
        for (int k = 0; k < NB; ++k) {
            const uint64_t s = k < 8 ? lo : hi;
            dst[k] = static_cast<uint8_t>(s >> ((k & 7) * 8));
        }
    }
}

template <int CPL, int W>
__device__ __forceinline__ void pack_row_w(uint8_t* row, int lane, uint64_t chunk) {
    if constexpr (W == 0) {
        return;
    } else {
        constexpr int G = 8 / CPL;          // lanes per 8 codes
        constexpr int CB = CPL * W;         // bits per lane (<= 64)
        uint64_t lo = chunk, hi = 0;
        // gather: stage s merges pairs at distance 2^s, doubling the bit count
#pragma unroll
        for (int s = 0, d = 1; d < G; ++s, d <<= 1) {
            const int sh = CB << s;         // bits held so far
            const uint64_t olo = __shfl_down_sync(kFull, lo, d);
            const uint64_t ohi = (2 * sh > 64) ? __shfl_down_sync(kFull, hi, d) : 0ull;
            if (sh < 64) {
                hi |= (olo >> (64 - sh)) | (ohi << sh);
                lo |= olo << sh;
            } else {
                hi |= olo;
            }
        }
        if ((lane % G) == 0) store_bytes<W, CPL == 4>(row + (lane / G) * W, lo, hi);
    }
}

// Store one row: `chunk` holds the lane's CPL codes, code c at bits [c w, c w + w).
template <int CPL>
__device__ __forceinline__ void pack_row(uint8_t* row, int lane, int w, uint64_t chunk) {
    switch (w) {
#define QS_W(N) case N: pack_row_w<CPL, N>(row, lane, chunk); break;
        QS_W(1) QS_W(2) QS_W(3) QS_W(4) QS_W(5) QS_W(6) QS_W(7) QS_W(8)
        QS_W(9) QS_W(10) QS_W(11) QS_W(12) QS_W(13) QS_W(14) QS_W(15) QS_W(16)
#undef QS_W
        default: break;
    }
}

// Issue the asynchronous copies of head g into stage S / payload buffer pay.  The head's
// payload window (in_off, in_end) and output offset come from the previous stage (or, for the
// first head, from direct loads); the window is checked before anything is copied.  One
// commit group per call.
template <int DK, int DV>
__device__ __noinline__ void wb_issue(WbStage<DK, DV>& S, uint8_t* pay, int g, int in_off, int in_end,
                                      int out_off, const WbParams& wp) {
    const StepParams& p = wp.s;
    const int tid = threadIdx.x;
    const bool stats = p.ema_s != nullptr;
    const int T = p.T;
        const int b = g / p.H, h = g - (g / p.H) * p.H;
        const size_t tok = (static_cast<size_t>(b) * T + p.t_begin) * p.H + h;
        const size_t rb = static_cast<size_t>(g) * DK;
        // fixed-size arrays, 16-byte chunks
        constexpr int C8 = DK / 16, C16 = DK * 2 / 16, C32 = DK * 4 / 16, CV = DV * 4 / 16;
        int c = tid;
        if (c < C8) cp_async16(S.w_in + 16 * c, p.in_widths + rb + 16 * c);
        else if ((c -= C8) < C8) cp_async16(S.w_out + 16 * c, p.out_widths + rb + 16 * c);
        else if ((c -= C8) < C8) cp_async16(S.fidx + 16 * c, p.in_fidx + rb + 16 * c);
        else if ((c -= C8) < C16) cp_async16(reinterpret_cast<uint8_t*>(S.sc_in) + 16 * c,
                                             reinterpret_cast<const uint8_t*>(p.in_scales + rb) + 16 * c);
        else if ((c -= C16) < C32) cp_async16(reinterpret_cast<uint8_t*>(S.k) + 16 * c,
                                              reinterpret_cast<const uint8_t*>(p.k + tok * DK) + 16 * c);
        else if ((c -= C32) < C32) cp_async16(reinterpret_cast<uint8_t*>(S.q) + 16 * c,
                                              reinterpret_cast<const uint8_t*>(p.q + tok * DK) + 16 * c);
        else if ((c -= C32) < CV) cp_async16(reinterpret_cast<uint8_t*>(S.v) + 16 * c,
                                             reinterpret_cast<const uint8_t*>(p.v + tok * DV) + 16 * c);
        else if ((c -= CV) < C32) {
            if (stats) cp_async16(reinterpret_cast<uint8_t*>(S.ms) + 16 * c,
                                  reinterpret_cast<const uint8_t*>(p.ema_s + rb) + 16 * c);
        } else if ((c -= C32) < C32) {
            if (stats) cp_async16(reinterpret_cast<uint8_t*>(S.mr) + 16 * c,
                                  reinterpret_cast<const uint8_t*>(p.ema_r + rb) + 16 * c);
        } else if ((c -= C32) < C32) {
            if (p.decay_row && !p.s_code) cp_async16(reinterpret_cast<uint8_t*>(S.s) + 16 * c,
                                                     reinterpret_cast<const uint8_t*>(p.s + tok * DK) + 16 * c);
        } else if ((c -= C32) < C8) {
            if (p.decay_row && p.s_code) cp_async16(S.scode + 16 * c, p.s_code + tok * DK + 16 * c);
        }
        // scalars and the offsets of the head after this one
        const int gn = g + gridDim.x;
        if (tid == 255) {
            if (p.erase) cp_async4(&S.beta, p.beta + tok);
            if (!p.decay_row && !p.s_code) cp_async4(&S.rate_h, p.s + tok);
        }
        if (tid == 254 && gn < wp.nheads) {
            const int hn = gn - (gn / p.H) * p.H;
            cp_async4(&S.nxt_in_off, p.in_head_off + gn);
            cp_async4(&S.nxt_out_off, p.out_head_off + gn);
            if (hn < p.H - 1) cp_async4(&S.nxt_in_end, p.in_head_off + gn + 1);
        }
        // payload window
        const int align = DV == 128 ? 16 : 8;
        const int nbytes = in_end - in_off;
        const bool ok = in_off >= 0 && nbytes >= 0 && nbytes <= p.stage_bytes && in_off % align == 0 &&
                        nbytes % align == 0 && static_cast<long long>(in_end) <= p.region_bytes;
        if (tid == 0) {
            S.in_off = in_off;
            S.in_end = in_end;
            S.out_off = out_off;
            S.ok = ok ? 1 : 0;
            // the following head's window ends at the next head's offset (copied above), or at
            // the end of the region for the last head of a batch element
            if (gn < wp.nheads && gn - (gn / p.H) * p.H == p.H - 1)
                S.nxt_in_end = static_cast<int>(p.region_bytes);
        }
        if (ok) {
            const uint8_t* src = p.in_payload + static_cast<size_t>(b) * p.region_bytes + in_off;
            if (DV == 128) {
                for (int i = tid; i < nbytes / 16; i += blockDim.x) cp_async16(pay + 16 * i, src + 16 * i);
            } else {
                for (int i = tid; i < nbytes / 8; i += blockDim.x) cp_async8(pay + 8 * i, src + 8 * i);
            }
        }
        cp_async_commit();
    }

// ---- the kernel ---------------------------------------------------------------------------------
template <int DK, int DV, int NW>
__global__ void __launch_bounds__(NW * 32, 1) wb_row_kernel(const WbParams wp) {
    constexpr int NT = NW * 32, RPW = DK / NW, CPL = DV / 32, CP2 = CPL / 2;
    constexpr int LOGR = RPW == 16 ? 4 : RPW == 8 ? 3 : RPW == 4 ? 2 : 1;
    using Sm = WbSmem<DK, DV, NW>;
    using Stage = WbStage<DK, DV>;
    static_assert(RPW >= 2 && RPW <= 16, "rows per warp");
    const StepParams& p = wp.s;
    extern __shared__ __align__(16) uint8_t smem_raw[];
    Sm& sm = *reinterpret_cast<Sm*>(smem_raw);
    const int pstride = (p.stage_bytes + 32 + 15) & ~15;
    uint8_t* pay0 = smem_raw + sizeof(Sm);
    uint8_t* pout = pay0 + 2 * pstride;
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const bool stats = p.ema_s != nullptr;
    const int T = p.T;

    if (tid < kNFit) sm.fitf[tid] = fit_factor(tid);
    if (tid >= 32 && tid < 32 + 17) {
        const int w = tid - 32;
        const float n = w >= 2 ? static_cast<float>((1 << (w - 1)) - 1) : 0.0f;
        sm.wc[w] = make_float4(n, w >= 2 ? __frcp_rn(n) : 0.0f, kMagic - n, kMagic + n);
    }

    const int g0 = blockIdx.x;
    if (g0 >= wp.nheads) return;
    {
        const int h0 = g0 % p.H;
        const int io = static_cast<int>(p.in_head_off[g0]);
        const int ie = h0 < p.H - 1 ? static_cast<int>(p.in_head_off[g0 + 1]) : static_cast<int>(p.region_bytes);
        const int oo = static_cast<int>(p.out_head_off[g0]);
        wb_issue<DK, DV>(sm.st[0], pay0, g0, io, ie, oo, wp);
    }

    for (int j = 0;; ++j) {
        const int g = g0 + j * gridDim.x;
        if (g >= wp.nheads) break;
        const int sidx = j & 1;
        Stage& S = sm.st[sidx];
        const uint8_t* pay = pay0 + sidx * pstride;
        const int b = g / p.H, h = g - (g / p.H) * p.H;
        cp_async_wait_all();
        if (tid == 0) sm.flag = S.ok ? 0 : 1;
        __syncthreads();                                                               // B1
        const int gn = g + gridDim.x;
        if (gn < wp.nheads)
            wb_issue<DK, DV>(sm.st[sidx ^ 1], pay0 + (sidx ^ 1) * pstride, gn, S.nxt_in_off, S.nxt_in_end,
                             S.nxt_out_off, wp);

        // ---- prep ---------------------------------------------------------------------------
        const size_t tok0 = (static_cast<size_t>(b) * T + p.t_begin) * p.H + h;
        const float beta0 = p.erase ? S.beta : 1.0f;
        float rate_h = 0.0f;
        if (!p.decay_row)
            rate_h = p.s_code ? __ldg(p.s_lut + static_cast<size_t>(h) * p.L +
                                      min(static_cast<int>(p.s_code[tok0]), p.L - 1))
                              : S.rate_h;
        if (warp < 2) {
            const uint8_t* wa = warp == 0 ? S.w_in : S.w_out;
            int* off = warp == 0 ? sm.off_in : sm.off_out;
            constexpr int PER = DK / 32;
            int loc[PER];
            int sum = 0;
            bool bad = false;
#pragma unroll
            for (int jj = 0; jj < PER; ++jj) {
                const int w = wa[lane * PER + jj];
                bad |= (w > 16);
                loc[jj] = sum;
                sum += w * (DV / 8);
            }
            int incl = sum;
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                const int n = __shfl_up_sync(kFull, incl, o);
                if (lane >= o) incl += n;
            }
#pragma unroll
            for (int jj = 0; jj < PER; ++jj) off[lane * PER + jj] = incl - sum + loc[jj];
            const int total = __shfl_sync(kFull, incl, 31);
            bad = __any_sync(kFull, bad);
            if (lane == 0) {
                off[DK] = total;
                const int align = DV == 128 ? 16 : 8;
                if (warp == 0) bad |= (total != S.in_end - S.in_off);
                else bad |= (total > p.stage_bytes || S.out_off % align != 0 || S.out_off < 0 ||
                             static_cast<long long>(S.out_off) + total > p.region_bytes);
                if (bad) atomicExch(&sm.flag, 1);
            }
        } else if (tid >= 64 && tid < 64 + DK) {
            const int i = tid - 64;
            const float kk = S.k[i];
            float rate = rate_h;
            if (p.decay_row)
                rate = p.s_code ? __ldg(p.s_lut + (static_cast<size_t>(h) * DK + i) * p.L +
                                        min(static_cast<int>(S.scode[i]), p.L - 1))
                                : S.s[i];
            if (!(rate > 0.0f) || !(rate < INFINITY)) raise_status(p.status, QS_DEV_RATE);
            const float d = expf(-rate);
            if (stats) {
                const float xs = -expm1f(-2.0f * rate);
                const float xr = p.erase ? __fmul_rn(__fmul_rn(beta0, __fsub_rn(2.0f, beta0)), __fmul_rn(kk, kk)) : 0.0f;
                if (p.t_begin == 0) {
                    S.ms[i] = xs;
                    S.mr[i] = xr;
                } else {
                    S.ms[i] = __fadd_rn(S.ms[i], __fmul_rn(p.alpha, __fsub_rn(xs, S.ms[i])));
                    S.mr[i] = __fadd_rn(S.mr[i], __fmul_rn(p.alpha, __fsub_rn(xr, S.mr[i])));
                }
            }
            const int w = min(static_cast<int>(S.w_in[i]), 16);
            const float D = f16_value(S.sc_in[i]);
            const float A = 8388608.0f + (w >= 2 ? sm.wc[w].x : 0.0f);
            sm.deq[i] = make_float4(-A, (w >= 2 ? D : (w == 1 ? -2.0f * D : 0.0f)) * d,
                                    (w == 1 ? D : 0.0f) * d, 0.0f);
            sm.a[i] = __fmul_rn(beta0, kk);
        } else if (tid >= 64 + DK && tid < 128 + DK) {
            // k . q over DK rows: 64 threads, DK / 64 rows each
            float kq = 0.0f;
#pragma unroll
            for (int r = tid - 64 - DK; r < DK; r += 64) kq = fmaf(S.k[r], S.q[r], kq);
            kq = warp_sum(kq);
            if (lane == 0) sm.wsum[(tid - 64 - DK) >> 5] = kq;
        }
        __syncthreads();                                                               // B2
        if (sm.flag != 0) {
            if (tid == 0) raise_status(p.status, QS_DEV_LAYOUT);
            continue;
        }

        // ---- unpack + dequantise (first token's decay folded in) -------------------------------
        float2 x[RPW][CP2];
#pragma unroll
        for (int r = 0; r < RPW; ++r) {
            const int i = warp * RPW + r;
            uint32_t u[CPL];
            extract_codes<CPL>(pay + sm.off_in[i], lane, S.w_in[i], u);
            const float4 dq = sm.deq[i];
            const float2 A2 = make_float2(dq.x, dq.x), S2 = make_float2(dq.y, dq.y), B2 = make_float2(dq.z, dq.z);
#pragma unroll
            for (int c = 0; c < CP2; ++c) {
                const float2 t = make_float2(__uint_as_float(kTwo23Bits | u[2 * c]),
                                             __uint_as_float(kTwo23Bits | u[2 * c + 1]));
                x[r][c] = __ffma2_rn(__fadd2_rn(t, A2), S2, B2);
            }
        }

        // ---- tokens of the interval (Eq. 1) ----------------------------------------------------
        for (int t = p.t_begin; t < p.t_end; ++t) {
            const size_t tok = (static_cast<size_t>(b) * T + t) * p.H + h;
            const float* kv = S.k;
            const float* qv = S.q;
            const float* vv = S.v;
            float beta = beta0;
            float kq;
            if (t > p.t_begin) {
                __syncthreads();   // every warp is done with the previous token's k and u
                beta = p.erase ? __ldg(p.beta + tok) : 1.0f;
                float rh = 0.0f;
                if (!p.decay_row)
                    rh = p.s_code ? __ldg(p.s_lut + static_cast<size_t>(h) * p.L +
                                          min(static_cast<int>(p.s_code[tok]), p.L - 1))
                                  : __ldg(p.s + tok);
                if (tid < DK) {
                    const int i = tid;
                    const float kk = __ldg(p.k + tok * DK + i), qq = __ldg(p.q + tok * DK + i);
                    sm.tk[i] = kk;
                    sm.tq[i] = qq;
                    float rate = rh;
                    if (p.decay_row)
                        rate = p.s_code ? __ldg(p.s_lut + (static_cast<size_t>(h) * DK + i) * p.L +
                                                min(static_cast<int>(p.s_code[tok * DK + i]), p.L - 1))
                                        : __ldg(p.s + tok * DK + i);
                    if (!(rate > 0.0f) || !(rate < INFINITY)) raise_status(p.status, QS_DEV_RATE);
                    sm.d[i] = expf(-rate);
                    sm.a[i] = __fmul_rn(beta, kk);
                    if (stats) {
                        const float xs = -expm1f(-2.0f * rate);
                        const float xr = p.erase ? __fmul_rn(__fmul_rn(beta, __fsub_rn(2.0f, beta)), __fmul_rn(kk, kk)) : 0.0f;
                        S.ms[i] = __fadd_rn(S.ms[i], __fmul_rn(p.alpha, __fsub_rn(xs, S.ms[i])));
                        S.mr[i] = __fadd_rn(S.mr[i], __fmul_rn(p.alpha, __fsub_rn(xr, S.mr[i])));
                    }
                    const float s2 = warp_sum(kk * qq);
                    if (lane == 0) sm.wsum[warp] = s2;
                }
                if (tid < DV) sm.tv[tid] = __ldg(p.v + tok * DV + tid);
                __syncthreads();
                kv = sm.tk;
                qv = sm.tq;
                vv = sm.tv;
#pragma unroll
                for (int r = 0; r < RPW; ++r) {
                    const float dd = sm.d[warp * RPW + r];
                    const float2 d2 = make_float2(dd, dd);
#pragma unroll
                    for (int c = 0; c < CP2; ++c) x[r][c] = __fmul2_rn(x[r][c], d2);
                }
            }
            float2 pp[CP2], rr[CP2];
#pragma unroll
            for (int c = 0; c < CP2; ++c) pp[c] = rr[c] = make_float2(0.0f, 0.0f);
#pragma unroll
            for (int r = 0; r < RPW; ++r) {
                const int i = warp * RPW + r;
                const float2 a2 = make_float2(sm.a[i], sm.a[i]);
                const float2 q2 = make_float2(qv[i], qv[i]);
#pragma unroll
                for (int c = 0; c < CP2; ++c) {
                    pp[c] = __ffma2_rn(x[r][c], a2, pp[c]);
                    rr[c] = __ffma2_rn(x[r][c], q2, rr[c]);
                }
            }
#pragma unroll
            for (int c = 0; c < CP2; ++c) {
                reinterpret_cast<float2*>(&sm.red[0][warp][lane * CPL])[c] = pp[c];
                reinterpret_cast<float2*>(&sm.red[1][warp][lane * CPL])[c] = rr[c];
            }
            __syncthreads();                                                           // B3
            if (tid < DV) {
                const int jv = tid;
                float P = 0.0f, Rr = 0.0f;
#pragma unroll
                for (int w = 0; w < NW; ++w) {
                    P += sm.red[0][w][jv];
                    Rr += sm.red[1][w][jv];
                }
                kq = 0.0f;
                if (t > p.t_begin) {
#pragma unroll
                    for (int w = 0; w < DK / 32; ++w) kq += sm.wsum[w];
                } else {
                    kq = sm.wsum[0] + sm.wsum[1];
                }
                const float vj = vv[jv];
                const float uu = p.erase ? __fsub_rn(__fmul_rn(beta, vj), P) : vj;
                sm.u[jv] = uu;
                p.o[tok * DV + jv] = fmaf(uu, kq, Rr);
            }
            __syncthreads();                                                           // B4
#pragma unroll
            for (int r = 0; r < RPW; ++r) {
                const float ki = kv[warp * RPW + r];
                const float2 k2 = make_float2(ki, ki);
#pragma unroll
                for (int c = 0; c < CP2; ++c)
                    x[r][c] = __ffma2_rn(k2, reinterpret_cast<const float2*>(&sm.u[lane * CPL])[c], x[r][c]);
            }
        }

        // ---- write-back (warp-local until B5) ---------------------------------------------------
        const bool refit = (p.fit_every <= 1) || ((p.w_index + h) % p.fit_every == 0);
        // row ranges (and 1-bit sums)
#pragma unroll
        for (int r = 0; r < RPW; ++r) {
            const int i = warp * RPW + r;
            float amax = 0.0f, asum = 0.0f;
#pragma unroll
            for (int c = 0; c < CP2; ++c) {
                amax = fmaxf(amax, fmaxf(fabsf(x[r][c].x), fabsf(x[r][c].y)));
                asum += fabsf(x[r][c].x) + fabsf(x[r][c].y);
            }
            const float R = warp_absmax(amax);
            if (S.w_out[i] == 1) asum = warp_sum(asum);
            if (lane == 0) {
                sm.rowR[i] = R;
                sm.rowM[i] = asum;
            }
        }
        __syncwarp();
        // per-row steps (lane r <-> row r): 1-bit means, rows that keep their factor, zero rows
        float myD = 0.0f, myInv = 0.0f;
        if (lane < RPW) {
            const int i = warp * RPW + lane, w = S.w_out[i];
            const float R = sm.rowR[i];
            int fidx = S.fidx[i];
            if (w == 1) {
                myD = f16_round(__fdiv_rn(sm.rowM[i], static_cast<float>(DV)));
            } else if (w >= 2) {
                if (R == 0.0f) {
                    if (refit) fidx = kNFit - 1;
                } else if (!refit) {
                    myD = cand_step(sm.fitf[fidx], R, sm.wc[w].y);
                    myInv = step_rcp(myD);
                }
            }
            sm.out_fidx[i] = static_cast<uint8_t>(fidx);
            sm.out_scale[i] = f16_bits(myD);
        }
        if (refit) {
            // the 16 candidate steps of every row: RPW x 16 (row, candidate) pairs over 32 lanes
#pragma unroll
            for (int pr = lane; pr < RPW * kNFit; pr += 32) {
                const int i = warp * RPW + (pr >> 4), k = pr & 15;
                const int w = S.w_out[i];
                const float R = sm.rowR[i];
                const float Dk = (w >= 2 && R > 0.0f) ? cand_step(sm.fitf[k], R, sm.wc[w].y) : 0.0f;
                sm.cand[i][k][0] = Dk;
                sm.cand[i][k][1] = step_rcp(Dk);
            }
            __syncwarp();
            // squared-error search: candidates outer, rows inner; lane l ends with row
            // (l >> (5 - LOGR)) and keeps the running minimum (ties to the larger factor)
            float2 ax[RPW][CP2];
#pragma unroll
            for (int r = 0; r < RPW; ++r)
#pragma unroll
                for (int c = 0; c < CP2; ++c) ax[r][c] = make_float2(fabsf(x[r][c].x), fabsf(x[r][c].y));
            float bsse = INFINITY;
            int bk = 0;
            const float2 mg2 = make_float2(kMagic, kMagic), nmg2 = make_float2(-kMagic, -kMagic);
#pragma unroll 1
            for (int k = 0; k < kNFit; ++k) {
                float part[RPW];
#pragma unroll
                for (int r = 0; r < RPW; ++r) {
                    const int i = warp * RPW + r;
                    const float2 cd = *reinterpret_cast<const float2*>(&sm.cand[i][k][0]);
                    const float lim = sm.wc[S.w_out[i]].w;
                    const float2 inv2 = make_float2(cd.y, cd.y), nD2 = make_float2(-cd.x, -cd.x);
                    float2 acc = make_float2(0.0f, 0.0f);
#pragma unroll
                    for (int c = 0; c < CP2; ++c) {
                        float2 t = __ffma2_rn(ax[r][c], inv2, mg2);
                        t.x = fminf(t.x, lim);
                        t.y = fminf(t.y, lim);
                        const float2 e = __ffma2_rn(__fadd2_rn(t, nmg2), nD2, ax[r][c]);
                        acc = __ffma2_rn(e, e, acc);
                    }
                    part[r] = acc.x + acc.y;
                }
                const float tot = reduce_rows<RPW>(part, lane);
                if (tot <= bsse) {
                    bsse = tot;
                    bk = k;
                }
            }
            if ((lane & ((32 >> LOGR) - 1)) == 0) sm.best_k[warp * RPW + (lane >> (5 - LOGR))] = bk;
            __syncwarp();
        }
        // codes, folded into one 64-bit chunk per lane and row
#pragma unroll
        for (int r = 0; r < RPW; ++r) {
            const int i = warp * RPW + r;
            const int w = S.w_out[i];
            float D = __shfl_sync(kFull, myD, r), inv = __shfl_sync(kFull, myInv, r);
            uint32_t u[4] = {0u, 0u, 0u, 0u};
            if (w >= 2) {
                const float4 wc = sm.wc[w];
                if (refit && sm.rowR[i] > 0.0f) {
                    const int best = sm.best_k[i];
                    const float2 cd = *reinterpret_cast<const float2*>(&sm.cand[i][best][0]);
                    D = cd.x;
                    inv = cd.y;
                    if (lane == 0) {
                        sm.out_fidx[i] = static_cast<uint8_t>(best);
                        sm.out_scale[i] = f16_bits(D);
                    }
                }
                const float2 inv2 = make_float2(inv, inv), mg2 = make_float2(kMagic, kMagic);
                const uint32_t off = kMagicBits - static_cast<uint32_t>(wc.x);
#pragma unroll
                for (int c = 0; c < CP2; ++c) {
                    const float2 tq = __fadd2_rn(__fmul2_rn(x[r][c], inv2), mg2);
                    u[2 * c] = __float_as_uint(fminf(fmaxf(tq.x, wc.z), wc.w)) - off;
                    u[2 * c + 1] = __float_as_uint(fminf(fmaxf(tq.y, wc.z), wc.w)) - off;
                }
            } else if (w == 1) {
#pragma unroll
                for (int c = 0; c < CP2; ++c) {
                    u[2 * c] = x[r][c].x < 0.0f ? 1u : 0u;
                    u[2 * c + 1] = x[r][c].y < 0.0f ? 1u : 0u;
                }
            }
            uint64_t ch = 0;
#pragma unroll
            for (int c = 0; c < CPL; ++c) ch |= static_cast<uint64_t>(u[c]) << (c * w);
            sm.chunk[warp][r][lane] = make_uint2(static_cast<uint32_t>(ch), static_cast<uint32_t>(ch >> 32));
        }
        __syncwarp();
#pragma unroll 1
        for (int r = 0; r < RPW; ++r) {
            const int i = warp * RPW + r;
            const uint2 c2 = sm.chunk[warp][r][lane];
            pack_row<CPL>(pout + sm.off_out[i], lane, S.w_out[i], (static_cast<uint64_t>(c2.y) << 32) | c2.x);
        }
        __syncthreads();                                                               // B5
        // ---- stores -------------------------------------------------------------------------------
        const int nbytes = sm.off_out[DK];
        uint8_t* dst = p.out_payload + static_cast<size_t>(b) * p.region_bytes + S.out_off;
        if (DV == 128) {
            for (int i = tid; i < nbytes / 16; i += NT)
                reinterpret_cast<uint4*>(dst)[i] = reinterpret_cast<const uint4*>(pout)[i];
        } else {
            for (int i = tid; i < nbytes / 8; i += NT)
                reinterpret_cast<uint2*>(dst)[i] = reinterpret_cast<const uint2*>(pout)[i];
        }
        const size_t rb = static_cast<size_t>(g) * DK;
        if (tid < DK) {
            p.out_scales[rb + tid] = sm.out_scale[tid];
            p.out_fidx[rb + tid] = sm.out_fidx[tid];
            if (p.range) p.range[rb + tid] = sm.rowR[tid];
            if (stats) {
                p.ema_s[rb + tid] = S.ms[tid];
                p.ema_r[rb + tid] = S.mr[tid];
            }
        }
    }
}

template <int DK, int DV, int NW>
cudaError_t launch_wb_row_t(const qstate_cfg& cfg, const StepParams& sp, cudaStream_t stream) {
    auto kern = wb_row_kernel<DK, DV, NW>;
    WbParams wp;
    wp.s = sp;
    wp.s.stage_bytes = DK * DV * cfg.bmax / 8;
    wp.nheads = cfg.B * cfg.H;
    const int pstride = (wp.s.stage_bytes + 32 + 15) & ~15;
    const size_t smem = sizeof(WbSmem<DK, DV, NW>) + 3 * static_cast<size_t>(pstride);
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         static_cast<int>(smem));
    if (e != cudaSuccess) return e;
    int dev = 0, sms = 0, per_sm = 0;
    if ((e = cudaGetDevice(&dev)) != cudaSuccess) return e;
    if ((e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess) return e;
    if ((e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, NW * 32, smem)) != cudaSuccess) return e;
    const int grid = std::min(wp.nheads, std::max(1, per_sm) * sms);
    kern<<<grid, NW * 32, smem, stream>>>(wp);
    return cudaGetLastError();
}

}  // namespace qs
