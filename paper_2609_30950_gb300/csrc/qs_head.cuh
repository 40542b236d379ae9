// qs_head.cuh -- write-back kernel for the head allocation unit (sm_103a): one width per head and
// one FP16 step per scale group of 32 key rows x 1 value column (Sec. 3, "Allocation units";
// Gated DeltaNet).  Also serves pack (dense -> packed) and unpack (packed -> dense) for this unit;
// the dense reference path runs the general kernel.
//
// One CTA of NW warps per (batch element, head).  Warp w owns row block w / NCS (32 key rows,
// exactly one scale-group row) and column slice w % NCS (CS value columns); lane l owns the CPL
// columns cs CS + l CPL .. + CPL - 1 of those 32 rows.  So every scale group lies in one lane,
// whole: its range, its 1-bit mean and the squared errors of its 16 candidate steps are
// register loops without any exchange, the candidate search is pruned per group, and with
// CPL = 2 the lane's two groups share packed FP32 instructions (`fma.rn.f32x2`), their
// per-group constants forming the operand pairs.  The head's FP32 state stays in registers:
//   1. widths (one per head) and layout checks; the head's packed rows are staged in shared
//      memory;
//   2. unpack + dequantise: x = (2^23 + u - (2^23 + n)) Delta d for the lane's groups;
//   3. per token (Eq. 1): decay, partials p = a^T S', r = q^T S' over the block's rows, column
//      sums across the DK/32 blocks in shared memory, u = w o v - p, o = r + u (k . q) (read
//      before quantising, Sec. 2), head statistics (Sec. 3), S += k u^T;
//   4. write-back: per group R = max |x|, then from f = 1 down the candidates' squared errors
//      until the clipping error of the group's maximum rules out the rest (exact: the result is
//      the exhaustive argmin), codes OR-ed into a zeroed shared staging region, one vector copy
//      of the region and coalesced stores of steps and factor indices.
#pragma once

#include <algorithm>
#include <type_traits>

#include "qs_common.cuh"

namespace qs {

template <int DK, int DV>
struct HeadGeom {
    static constexpr int CPL = (DK >= 128 && DV >= 128) ? 2 : 1;   // value columns per lane
    static constexpr int NB = DK / 32;     // row blocks (one scale-group row each)
    static constexpr int CS = 32 * CPL;    // value columns per slice (one warp)
    static constexpr int NCS = DV / CS;    // column slices per row block
    static constexpr int NW = NB * NCS;    // warps: 8 at 128 x 128 and 128 x 64, 4 at 64 x 64
    static constexpr int NT = 32 * NW;
    static constexpr int NSG = NB * DV;    // scale groups per head
    static constexpr bool ok = DK % 32 == 0 && DV % CS == 0 && NW <= 8 && DK <= NT && DV < NT;
};

template <int DK, int DV>
struct alignas(16) HeadSmem {
    using G = HeadGeom<DK, DV>;
    float4 aq[DK];             // (a_i, a_i, q_i, q_i): erase vector and query as operand pairs
    float2 kk[DK];             // (k_i, k_i)
    float v[DV], u[DV], gw[DV];
    float red[2][G::NB][DV];   // p and r partials per row block
    float wsum[4][DK / 32];    // per-warp k.q, |k|^2, a.k, |a|^2
    float fitf[kNFit];         // f_k = (5 + k) / 20
    float ms, mr;              // head statistics (Sec. 3)
};

// One lane's values of one row: CPL columns, packed when CPL = 2.
template <int CPL> struct HeadLane;
template <> struct HeadLane<2> { using V = float2; };
template <> struct HeadLane<1> { using V = float; };

__device__ __forceinline__ float2 hv_fma(float2 a, float2 b, float2 c) { return __ffma2_rn(a, b, c); }
__device__ __forceinline__ float hv_fma(float a, float b, float c) { return __fmaf_rn(a, b, c); }
__device__ __forceinline__ float2 hv_mul(float2 a, float2 b) { return __fmul2_rn(a, b); }
__device__ __forceinline__ float hv_mul(float a, float b) { return __fmul_rn(a, b); }
__device__ __forceinline__ float2 hv_add(float2 a, float2 b) { return __fadd2_rn(a, b); }
__device__ __forceinline__ float hv_add(float a, float b) { return __fadd_rn(a, b); }
template <class V> __device__ __forceinline__ V hv_bc(float s);
template <> __device__ __forceinline__ float2 hv_bc<float2>(float s) { return make_float2(s, s); }
template <> __device__ __forceinline__ float hv_bc<float>(float s) { return s; }
__device__ __forceinline__ float hv_get(float2 v, int c) { return c == 0 ? v.x : v.y; }
__device__ __forceinline__ float hv_get(float v, int) { return v; }
__device__ __forceinline__ void hv_set(float2& v, int c, float s) { if (c == 0) v.x = s; else v.y = s; }
__device__ __forceinline__ void hv_set(float& v, int, float s) { v = s; }
__device__ __forceinline__ float2 hv_abs(float2 v) { return make_float2(fabsf(v.x), fabsf(v.y)); }
__device__ __forceinline__ float hv_abs(float v) { return fabsf(v); }

template <int DK, int DV, bool SRC_PACKED, bool DST_PACKED>
__global__ void __launch_bounds__(HeadGeom<DK, DV>::NT, 2) head_kernel(const StepParams p) {
    using G = HeadGeom<DK, DV>;
    static_assert(G::ok, "head-unit layout");
    constexpr int NB = G::NB, NCS = G::NCS, CS = G::CS, CPL = G::CPL, NSG = G::NSG, NT = G::NT;
    using V = typename HeadLane<CPL>::V;
    using Sm = HeadSmem<DK, DV>;
    extern __shared__ __align__(16) uint8_t smem_raw[];
    Sm& sm = *reinterpret_cast<Sm*>(smem_raw);
    uint8_t* pay = smem_raw + sizeof(Sm);

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int bh = blockIdx.x, b = bh / p.H, h = bh - b * p.H;
    const int blk = warp / NCS, cs = warp - blk * NCS;
    const int r0 = 32 * blk;                 // the lane's first key row
    const int col0 = cs * CS + lane * CPL;   // the lane's first value column
    const size_t gbase = static_cast<size_t>(bh) * NSG + static_cast<size_t>(blk) * DV + col0;
    const bool has_tokens = p.t_end > p.t_begin;
    const bool stats = has_tokens && p.ema_s != nullptr;
    constexpr int align = DV == 128 ? 16 : 8;

    // ---- 1. widths and layout ---------------------------------------------------------------
    const int w_in = SRC_PACKED ? static_cast<int>(p.in_widths[bh]) : 0;
    const int w_out = DST_PACKED ? static_cast<int>(p.out_widths[bh]) : 0;
    const int bytes_in = DK * DV / 8 * w_in, bytes_out = DK * DV / 8 * w_out;
    bool bad = false;
    if (SRC_PACKED) {
        const long long o = p.in_head_off[bh];
        bad |= w_in > 16 || o % align != 0 || o + bytes_in > p.region_bytes || bytes_in > p.stage_bytes;
    }
    if (DST_PACKED) {
        const long long o = p.out_head_off[bh];
        bad |= w_out > 16 || o % align != 0 || o + bytes_out > p.region_bytes || bytes_out > p.stage_bytes;
    }
    if (bad) {   // uniform over the CTA: nothing has been written yet
        if (tid == 0) raise_status(p.status, QS_DEV_LAYOUT);
        return;
    }
    using Vec = typename std::conditional<DV == 128, uint4, uint2>::type;
    if (SRC_PACKED) {
        const Vec* src = reinterpret_cast<const Vec*>(p.in_payload + static_cast<size_t>(b) * p.region_bytes +
                                                      p.in_head_off[bh]);
        Vec* dst = reinterpret_cast<Vec*>(pay);
        for (int i = tid; i < bytes_in / static_cast<int>(sizeof(Vec)); i += NT) dst[i] = __ldg(src + i);
        if (tid < 4) reinterpret_cast<uint32_t*>(pay + bytes_in)[tid] = 0u;   // readable tail
    }
    if (tid < kNFit) sm.fitf[tid] = fit_factor(tid);
    if (stats && tid == 0) {
        sm.ms = p.ema_s[bh];
        sm.mr = p.ema_r[bh];
    }
    __syncthreads();

    // ---- 2. unpack + dequantise ---------------------------------------------------------------
    V x[32];
    if (SRC_PACKED) {
        // per group: x = ((2^23 + u) - (2^23 + n)) Delta (w >= 2), (1 - 2u) m (w = 1), 0 (w = 0)
        const float nA = -(8388608.0f + (w_in >= 2 ? static_cast<float>((1 << (w_in - 1)) - 1) : 0.0f));
        V S2, B2;
#pragma unroll
        for (int c = 0; c < CPL; ++c) {
            const float D = f16_value(p.in_scales[gbase + c]);
            hv_set(S2, c, w_in >= 2 ? D : (w_in == 1 ? -2.0f * D : 0.0f));
            hv_set(B2, c, w_in == 1 ? D : 0.0f);
        }
        const V A2 = hv_bc<V>(nA);
        const int rowbytes = w_in * (DV / 8);
        const int P = col0 * w_in, idx = P >> 5, sh = P & 31;
        const uint32_t mask = (1u << w_in) - 1u;
        const uint8_t* base = pay + r0 * rowbytes + 4 * idx;
#pragma unroll
        for (int r = 0; r < 32; ++r) {
            const uint32_t* wd = reinterpret_cast<const uint32_t*>(base + r * rowbytes);
            const uint32_t chunk = w_in == 0 ? 0u : __funnelshift_r(wd[0], wd[1], sh);
            V t;
#pragma unroll
            for (int c = 0; c < CPL; ++c) hv_set(t, c, __uint_as_float(kTwo23Bits | ((chunk >> (c * w_in)) & mask)));
            x[r] = hv_fma(hv_add(t, A2), S2, B2);
        }
    } else if (p.dense_in != nullptr) {
        const float* src = p.dense_in + (static_cast<size_t>(bh) * DK + r0) * DV + col0;
#pragma unroll
        for (int r = 0; r < 32; ++r) {
            if constexpr (CPL == 2) x[r] = *reinterpret_cast<const float2*>(src + r * DV);
            else x[r] = src[r * DV];
        }
    } else {
#pragma unroll
        for (int r = 0; r < 32; ++r) x[r] = hv_bc<V>(0.0f);
    }
    if (SRC_PACKED) __syncthreads();   // the staging buffer is reused for the output rows
    if (DST_PACKED) {                  // zero the output rows: codes are OR-ed in
        const int nz = (bytes_out + 16) / 16;
        for (int i = tid; i < nz; i += NT) reinterpret_cast<uint4*>(pay)[i] = make_uint4(0, 0, 0, 0);
        if (!has_tokens) __syncthreads();
    }

    // ---- 3. tokens of this write-back interval (Eq. 1) ------------------------------------------
    for (int t = p.t_begin; t < p.t_end; ++t) {
        if (t > p.t_begin) __syncthreads();   // every warp is done with the previous token's k, u
        const size_t tok = (static_cast<size_t>(b) * p.T + t) * p.H + h;
        const float beta = p.erase ? __ldg(p.beta + tok) : 1.0f;
        const float rate = p.s_code ? __ldg(p.s_lut + static_cast<size_t>(h) * p.L +
                                            min(static_cast<int>(p.s_code[tok]), p.L - 1))
                                    : __ldg(p.s + tok);
        if (tid == 0 && (!(rate > 0.0f) || !(rate < INFINITY))) raise_status(p.status, QS_DEV_RATE);
        if (tid < DK) {
            const int i = tid;
            const float kk = __ldg(p.k + tok * DK + i), qq = __ldg(p.q + tok * DK + i);
            const float ai = p.general ? __ldg(p.a_in + tok * DK + i) : __fmul_rn(beta, kk);
            sm.aq[i] = make_float4(ai, ai, qq, qq);
            sm.kk[i] = make_float2(kk, kk);
            const float kq = warp_sum(kk * qq);
            const float k2 = warp_sum(kk * kk);
            float ak = 0.0f, aa = 0.0f;
            if (p.general) {
                ak = warp_sum(ai * kk);
                aa = warp_sum(ai * ai);
            }
            if (lane == 0) {
                sm.wsum[0][warp] = kq;
                sm.wsum[1][warp] = k2;
                sm.wsum[2][warp] = ak;
                sm.wsum[3][warp] = aa;
            }
        }
        if (tid < DV) {
            sm.v[tid] = __ldg(p.v + tok * DV + tid);
            if (p.general) sm.gw[tid] = __ldg(p.w_in + tok * DV + tid);
        }
        __syncthreads();
        // decay and partials over the block's rows
        const V d2 = hv_bc<V>(expf(-rate));
        V pp = hv_bc<V>(0.0f), rr = hv_bc<V>(0.0f);
#pragma unroll
        for (int r = 0; r < 32; ++r) {
            const float4 aq = sm.aq[r0 + r];
            x[r] = hv_mul(x[r], d2);
            if constexpr (CPL == 2) {
                pp = hv_fma(x[r], make_float2(aq.x, aq.y), pp);
                rr = hv_fma(x[r], make_float2(aq.z, aq.w), rr);
            } else {
                pp = hv_fma(x[r], aq.x, pp);
                rr = hv_fma(x[r], aq.z, rr);
            }
        }
#pragma unroll
        for (int c = 0; c < CPL; ++c) {
            sm.red[0][blk][col0 + c] = hv_get(pp, c);
            sm.red[1][blk][col0 + c] = hv_get(rr, c);
        }
        __syncthreads();
        if (tid < DV) {
            const int j = tid;
            float P = 0.0f, Rr = 0.0f, kq = 0.0f;
#pragma unroll
            for (int k = 0; k < NB; ++k) {
                P += sm.red[0][k][j];
                Rr += sm.red[1][k][j];
            }
#pragma unroll
            for (int w = 0; w < DK / 32; ++w) kq += sm.wsum[0][w];
            const float vj = sm.v[j];
            // S = S' - k (a^T S') + k (w o v)^T:  u = beta v - p (delta rule), u = v (no erase)
            const float wj = p.general ? sm.gw[j] : beta;
            const float u = (p.erase || p.general) ? __fsub_rn(__fmul_rn(wj, vj), P) : vj;
            sm.u[j] = u;
            p.o[tok * DV + j] = fmaf(u, kq, Rr);   // o = S^T q = S'^T q + u (k . q)
        }
        if (stats && tid == DV) {   // Sec. 3 statistics per head (a thread with no column)
            float k2 = 0.0f;
#pragma unroll
            for (int w = 0; w < DK / 32; ++w) k2 += sm.wsum[1][w];
            const float xs = -expm1f(-2.0f * rate);
            float xr = p.erase ? __fmul_rn(__fmul_rn(beta, __fsub_rn(2.0f, beta)),
                                           __fdiv_rn(k2, static_cast<float>(DK)))
                               : 0.0f;
            if (p.general) {   // mean over the rows of 2 a_i k_i - a_i^2 |k|^2
                float ak = 0.0f, aa = 0.0f;
#pragma unroll
                for (int w = 0; w < DK / 32; ++w) {
                    ak += sm.wsum[2][w];
                    aa += sm.wsum[3][w];
                }
                xr = __fdiv_rn(__fsub_rn(__fmul_rn(2.0f, ak), __fmul_rn(aa, k2)), static_cast<float>(DK));
            }
            if (t == 0) {
                sm.ms = xs;
                sm.mr = xr;
            } else {
                sm.ms = __fadd_rn(sm.ms, __fmul_rn(p.alpha, __fsub_rn(xs, sm.ms)));
                sm.mr = __fadd_rn(sm.mr, __fmul_rn(p.alpha, __fsub_rn(xr, sm.mr)));
            }
        }
        __syncthreads();
        V u2;
#pragma unroll
        for (int c = 0; c < CPL; ++c) hv_set(u2, c, sm.u[col0 + c]);
#pragma unroll
        for (int r = 0; r < 32; ++r) {
            if constexpr (CPL == 2) x[r] = hv_fma(sm.kk[r0 + r], u2, x[r]);
            else x[r] = hv_fma(sm.kk[r0 + r].x, u2, x[r]);
        }
    }

    // ---- 4. write-back ----------------------------------------------------------------------------
    if (DST_PACKED) {
        const int w = w_out;
        const bool refit = (p.fit_every <= 1) || ((p.w_index + h) % p.fit_every == 0);
        // magnitudes in place, signs kept aside (bit r of sg[c] = row r of column c negative)
        uint32_t sg[CPL];
        V Rg = hv_bc<V>(0.0f), Mg = hv_bc<V>(0.0f);
#pragma unroll
        for (int c = 0; c < CPL; ++c) sg[c] = 0u;
#pragma unroll
        for (int r = 0; r < 32; ++r) {
#pragma unroll
            for (int c = 0; c < CPL; ++c) {
                const float xv = hv_get(x[r], c), av = fabsf(xv);
                sg[c] |= (xv < 0.0f ? 1u : 0u) << r;
                hv_set(x[r], c, av);
                hv_set(Rg, c, fmaxf(hv_get(Rg, c), av));
                if (w == 1) hv_set(Mg, c, __fadd_rn(hv_get(Mg, c), av));   // in row order
            }
        }
        int fidx[CPL];
        float D[CPL];
        const float nf = w >= 2 ? static_cast<float>((1 << (w - 1)) - 1) : 0.0f;
        const float inv_n = w >= 2 ? __frcp_rn(nf) : 0.0f;
#pragma unroll
        for (int c = 0; c < CPL; ++c) {
            fidx[c] = p.in_fidx ? static_cast<int>(p.in_fidx[gbase + c]) : kNFit - 1;
            D[c] = 0.0f;
        }
        if (w == 1) {
#pragma unroll
            for (int c = 0; c < CPL; ++c) D[c] = f16_round(__fdiv_rn(hv_get(Mg, c), 32.0f));
        } else if (w >= 2 && refit) {
            // From f = 1 down: every element at or above n Delta_k quantises to n, so the clipping
            // error of the group's maximum bounds candidate k's error from below and grows as k
            // falls; once it exceeds the best error found (2^-10 margin for rounding) no smaller
            // factor can win.  Equal errors go to the larger factor.  The search takes approximate
            // reciprocals; the chosen step's IEEE reciprocal is taken for the codes.
            float best[CPL];
#pragma unroll
            for (int c = 0; c < CPL; ++c) {
                best[c] = INFINITY;
                fidx[c] = kNFit - 1;
            }
            const float lim = kMagic + nf;
            const V M2 = hv_bc<V>(kMagic), nM2 = hv_bc<V>(-kMagic);
            // Candidates k and k - 1 per round (independent work for the lane); the second is
            // evaluated even when its bound already rules it out, and then cannot win.
            auto cand = [&](int k, V& iv, V& nd) {
                const float f = sm.fitf[k];
#pragma unroll
                for (int c = 0; c < CPL; ++c) {
                    const float R = hv_get(Rg, c);
                    const float Dk = R > 0.0f ? cand_step(f, R, inv_n) : 0.0f;
                    float ik = 0.0f;
                    if (Dk > 0.0f) asm("rcp.approx.ftz.f32 %0, %1;" : "=f"(ik) : "f"(Dk));
                    hv_set(iv, c, ik);
                    hv_set(nd, c, -Dk);
                }
            };
#pragma unroll 1
            for (int k = kNFit - 1; k >= 0; k -= 2) {
                const int kb = k >= 1 ? k - 1 : k;
                V ivA, ndA, ivB, ndB;
                cand(k, ivA, ndA);
                cand(kb, ivB, ndB);
                bool go[CPL], any = false;
#pragma unroll
                for (int c = 0; c < CPL; ++c) {
                    const float R = hv_get(Rg, c);
                    const float e = fmaxf(R + nf * hv_get(ndA, c), 0.0f);
                    go[c] = R > 0.0f && e * e <= best[c] * (1.0f + 1.0f / 1024.0f);
                    any |= go[c];
                }
                if (!__any_sync(kFull, any)) break;
                V aA = hv_bc<V>(0.0f), aB = hv_bc<V>(0.0f);
#pragma unroll
                for (int r = 0; r < 32; ++r) {
                    V tA = hv_fma(x[r], ivA, M2), tB = hv_fma(x[r], ivB, M2);
#pragma unroll
                    for (int c = 0; c < CPL; ++c) {
                        hv_set(tA, c, fminf(hv_get(tA, c), lim));
                        hv_set(tB, c, fminf(hv_get(tB, c), lim));
                    }
                    const V eA = hv_fma(hv_add(tA, nM2), ndA, x[r]);
                    const V eB = hv_fma(hv_add(tB, nM2), ndB, x[r]);
                    aA = hv_fma(eA, eA, aA);
                    aB = hv_fma(eB, eB, aB);
                }
#pragma unroll
                for (int c = 0; c < CPL; ++c) {
                    if (go[c] && hv_get(aA, c) < best[c]) {
                        best[c] = hv_get(aA, c);
                        fidx[c] = k;
                    }
                    if (kb < k && hv_get(Rg, c) > 0.0f && hv_get(aB, c) < best[c]) {
                        best[c] = hv_get(aB, c);
                        fidx[c] = kb;
                    }
                }
            }
#pragma unroll
            for (int c = 0; c < CPL; ++c) {
                const float R = hv_get(Rg, c);
                if (R == 0.0f) fidx[c] = kNFit - 1;
                D[c] = R > 0.0f ? cand_step(sm.fitf[fidx[c]], R, inv_n) : 0.0f;
            }
        } else if (w >= 2) {
#pragma unroll
            for (int c = 0; c < CPL; ++c) {
                const float R = hv_get(Rg, c);
                D[c] = R > 0.0f ? cand_step(sm.fitf[fidx[c]], R, inv_n) : 0.0f;
            }
        }
        // codes (offset binary q + n; 1 bit: sign), OR-ed into the row at bit col0 w
        if (w >= 1) {
            V inv2;
#pragma unroll
            for (int c = 0; c < CPL; ++c) hv_set(inv2, c, step_rcp(D[c]));
            const int n = w >= 2 ? (1 << (w - 1)) - 1 : 0;
            const int rowbytes = w * (DV / 8);
            const int P = col0 * w, idx = P >> 5, sh = P & 31;
            uint32_t* words = reinterpret_cast<uint32_t*>(pay + r0 * rowbytes) + idx;
#pragma unroll
            for (int r = 0; r < 32; ++r) {
                uint32_t chunk = 0u;
                if (w >= 2) {
                    // restore the sign, then q = clamp(rint(x / Delta), -n, n) on the rounded bits
                    V xs;
#pragma unroll
                    for (int c = 0; c < CPL; ++c)
                        hv_set(xs, c, __uint_as_float(__float_as_uint(hv_get(x[r], c)) | (((sg[c] >> r) & 1u) << 31)));
                    const V tq = hv_add(hv_mul(xs, inv2), hv_bc<V>(kMagic));
#pragma unroll
                    for (int c = 0; c < CPL; ++c)
                        chunk |= static_cast<uint32_t>(__viaddmin_s32_relu(__float_as_int(hv_get(tq, c)),
                                                                           n - static_cast<int>(kMagicBits), 2 * n))
                                 << (c * w);
                } else {
#pragma unroll
                    for (int c = 0; c < CPL; ++c) chunk |= ((sg[c] >> r) & 1u) << c;
                }
                uint32_t* wd = reinterpret_cast<uint32_t*>(reinterpret_cast<uint8_t*>(words) + r * rowbytes);
                const uint64_t sh64 = static_cast<uint64_t>(chunk) << sh;
                const uint32_t lo = static_cast<uint32_t>(sh64), hi = static_cast<uint32_t>(sh64 >> 32);
                if (lo) atomicOr(wd, lo);
                if (hi) atomicOr(wd + 1, hi);
            }
        }
#pragma unroll
        for (int c = 0; c < CPL; ++c) {
            p.out_scales[gbase + c] = f16_bits(D[c]);
            p.out_fidx[gbase + c] = static_cast<uint8_t>(fidx[c]);
        }
        __syncthreads();
        Vec* dst = reinterpret_cast<Vec*>(p.out_payload + static_cast<size_t>(b) * p.region_bytes + p.out_head_off[bh]);
        const Vec* srcv = reinterpret_cast<const Vec*>(pay);
        for (int i = tid; i < bytes_out / static_cast<int>(sizeof(Vec)); i += NT) dst[i] = srcv[i];
    } else if (p.dense_out != nullptr) {
        float* dst = p.dense_out + (static_cast<size_t>(bh) * DK + r0) * DV + col0;
#pragma unroll
        for (int r = 0; r < 32; ++r) {
            if constexpr (CPL == 2) *reinterpret_cast<float2*>(dst + r * DV) = x[r];
            else dst[r * DV] = x[r];
        }
    }
    if (stats && tid == 0) {
        p.ema_s[bh] = sm.ms;
        p.ema_r[bh] = sm.mr;
    }
}

template <int DK, int DV, bool SRC_PACKED, bool DST_PACKED>
cudaError_t launch_head_t(const qstate_cfg& cfg, const StepParams& p, cudaStream_t stream) {
    auto kern = head_kernel<DK, DV, SRC_PACKED, DST_PACKED>;
    const int stage = DK * DV * cfg.bmax / 8;
    const size_t smem = sizeof(HeadSmem<DK, DV>) + static_cast<size_t>(stage) + 32;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         static_cast<int>(smem));
    if (e != cudaSuccess) return e;
    StepParams q = p;
    q.stage_bytes = stage;
    kern<<<cfg.B * cfg.H, HeadGeom<DK, DV>::NT, smem, stream>>>(q);
    return cudaGetLastError();
}

}  // namespace qs

namespace qs {

// Decoding and dequantisation of a head's rows at a compile-time width W (the persistent
// kernel switches once per head): the lane's CPL codes of row r sit at bit col0 W of the row, in
// one word when CPL W divides 32, else across two; x = (2^23 + u - A) S + B as in the kernel
// above.
template <int W, int DV, int CPL, class V>
__device__ __forceinline__ void head_unpack_rows(const uint8_t* pay, int r0, int col0, V A2, V S2, V B2,
                                                 V (&x)[32]) {
    if constexpr (W == 0) {
#pragma unroll
        for (int r = 0; r < 32; ++r) x[r] = hv_bc<V>(0.0f);
    } else {
        constexpr int rowbytes = W * (DV / 8);
        constexpr uint32_t mask = (1u << W) - 1u;
        const int P = col0 * W, idx = P >> 5, sh = P & 31;
        const uint8_t* base = pay + r0 * rowbytes + 4 * idx;
#pragma unroll
        for (int r = 0; r < 32; ++r) {
            const uint32_t* wd = reinterpret_cast<const uint32_t*>(base + r * rowbytes);
            uint32_t chunk;
            if constexpr (32 % (CPL * W) == 0) chunk = wd[0] >> sh;
            else chunk = __funnelshift_r(wd[0], wd[1], sh);
            V t;
#pragma unroll
            for (int c = 0; c < CPL; ++c) hv_set(t, c, __uint_as_float(kTwo23Bits | ((chunk >> (c * W)) & mask)));
            x[r] = hv_fma(hv_add(t, A2), S2, B2);
        }
    }
}

// Codes and packing of a head's rows (Sec. 3, "Levels and storage") at a compile-time width W
// (one width per head, so the kernel switches once per head): the lane's CPL codes of row r
// (offset binary for W >= 2; for W = 1 the sign bit, 1 for x < 0, negative zero counting as
// positive) are OR-ed into the row's bit stream at bit col0 W.  A lane's CPL W bits stay within
// one word when CPL W divides 32; at CPL W = 32 the word is the lane's alone.
template <int W, int DV, int CPL, class V>
__device__ __forceinline__ void head_pack_rows(const V (&x)[32], V inv2, uint8_t* pout, int r0, int col0) {
    constexpr int rowbytes = W * (DV / 8);
    constexpr int n = W >= 2 ? (1 << (W - 1)) - 1 : 0;
    const int P = col0 * W, idx = P >> 5, sh = P & 31;
    uint32_t* words = reinterpret_cast<uint32_t*>(pout + r0 * rowbytes) + idx;
#pragma unroll
    for (int r = 0; r < 32; ++r) {
        uint32_t chunk = 0u;
        if constexpr (W >= 2) {
            const V tq = hv_add(hv_mul(x[r], inv2), hv_bc<V>(kMagic));
#pragma unroll
            for (int c = 0; c < CPL; ++c)
                chunk |= static_cast<uint32_t>(__viaddmin_s32_relu(__float_as_int(hv_get(tq, c)),
                                                                   n - static_cast<int>(kMagicBits), 2 * n)) << (c * W);
        } else {
#pragma unroll
            for (int c = 0; c < CPL; ++c) chunk |= (hv_get(x[r], c) < 0.0f ? 1u : 0u) << c;
        }
        uint32_t* wd = reinterpret_cast<uint32_t*>(reinterpret_cast<uint8_t*>(words) + r * rowbytes);
        if constexpr (CPL * W == 32) {
            *wd = chunk;
        } else if constexpr (32 % (CPL * W) == 0) {
            if (chunk) atomicOr(wd, chunk << sh);
        } else {
            const uint64_t sh64 = static_cast<uint64_t>(chunk) << sh;
            const uint32_t lo = static_cast<uint32_t>(sh64), hi = static_cast<uint32_t>(sh64 >> 32);
            if (lo) atomicOr(wd, lo);
            if (hi) atomicOr(wd + 1, hi);
        }
    }
}

// ---- persistent write-back of the head unit ---------------------------------------------------
// The write-back kernel above (one CTA per head) loads a head's payload, steps and inputs only
// when the CTA starts, so every head begins with a wait on global memory.  This variant keeps
// NW-warp CTAs resident (two per SM) over a contiguous block of heads and copies head g + 1's
// packed rows, FP16 steps, fitted factors and first-token inputs into the other half of a double
// buffer with cp.async while head g computes; the widths and offsets that size those copies are
// read one head earlier still.  The head's codes are OR-ed into a separate output buffer.  The
// range-factor search evaluates one candidate per round with the 32 rows split over two
// accumulators (fewer live registers than candidate pairs, and no second candidate evaluated
// after the bound has ruled it out).  Unpack, tokens, codes and statistics are the kernel
// above's operations; the candidates' squared errors are summed in another order, so a fitted
// factor can differ from that kernel's only where two candidates tie within rounding.
template <int DK, int DV>
struct alignas(16) HeadStage {
    using G = HeadGeom<DK, DV>;
    float k[DK], q[DK], v[DV];      // the interval's first token
    uint16_t sc[G::NSG];            // FP16 steps of the input state's scale groups
    uint8_t fidx[G::NSG];           // fitted factors of the previous write-back
    float beta, rate, ms, mr;       // first token's beta and decay rate; head statistics
    int w_in, w_out, in_off, out_off;
    int ok, pad[3];
};

__device__ __forceinline__ void hd_cp16(void* smem, const void* gmem) {
    const unsigned s = static_cast<unsigned>(__cvta_generic_to_shared(smem));
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;\n" ::"r"(s), "l"(gmem) : "memory");
}
__device__ __forceinline__ void hd_cp8(void* smem, const void* gmem) {
    const unsigned s = static_cast<unsigned>(__cvta_generic_to_shared(smem));
    asm volatile("cp.async.ca.shared.global [%0], [%1], 8;\n" ::"r"(s), "l"(gmem) : "memory");
}
__device__ __forceinline__ void hd_commit() { asm volatile("cp.async.commit_group;\n" ::: "memory"); }
__device__ __forceinline__ void hd_wait_all() { asm volatile("cp.async.wait_group 0;\n" ::: "memory"); }

// Head bh's metadata (widths, payload offsets) and its layout check.
struct HeadMeta {
    int w_in, w_out, in_off, out_off, ok;
};
template <int DK, int DV>
__device__ __forceinline__ HeadMeta head_meta(const StepParams& p, int bh) {
    constexpr int align = DV == 128 ? 16 : 8;
    HeadMeta m;
    m.w_in = __ldg(p.in_widths + bh);
    m.w_out = __ldg(p.out_widths + bh);
    m.in_off = static_cast<int>(__ldg(p.in_head_off + bh));
    m.out_off = static_cast<int>(__ldg(p.out_head_off + bh));
    const long long bi = static_cast<long long>(DK) * DV / 8 * m.w_in, bo = static_cast<long long>(DK) * DV / 8 * m.w_out;
    m.ok = !(m.w_in > 16 || m.in_off < 0 || m.in_off % align != 0 || m.in_off + bi > p.region_bytes ||
             bi > p.stage_bytes || m.w_out > 16 || m.out_off < 0 || m.out_off % align != 0 ||
             m.out_off + bo > p.region_bytes || bo > p.stage_bytes);
    return m;
}

// Copies of head bh's inputs into stage S and payload buffer pay (all threads; one commit group).
template <int DK, int DV>
__device__ __forceinline__ void head_issue(HeadStage<DK, DV>& S, uint8_t* pay, const HeadMeta& m, int bh,
                                           const StepParams& p) {
    using G = HeadGeom<DK, DV>;
    const int tid = threadIdx.x;
    const int b = bh / p.H;
    if (m.ok) {
        const int nbytes = DK * DV / 8 * m.w_in;
        const uint8_t* src = p.in_payload + static_cast<size_t>(b) * p.region_bytes + m.in_off;
        if (DV == 128) {
            for (int i = tid; i < nbytes / 16; i += G::NT) hd_cp16(pay + 16 * i, src + 16 * i);
        } else {
            for (int i = tid; i < nbytes / 8; i += G::NT) hd_cp8(pay + 8 * i, src + 8 * i);
        }
        const uint8_t* sc = reinterpret_cast<const uint8_t*>(p.in_scales + static_cast<size_t>(bh) * G::NSG);
        for (int i = tid; i < G::NSG * 2 / 16; i += G::NT) hd_cp16(reinterpret_cast<uint8_t*>(S.sc) + 16 * i, sc + 16 * i);
        const uint8_t* fi = p.in_fidx + static_cast<size_t>(bh) * G::NSG;
        for (int i = tid; i < G::NSG / 16; i += G::NT) hd_cp16(S.fidx + 16 * i, fi + 16 * i);
        if (p.t_end > p.t_begin) {
            const int h = bh - b * p.H;
            const size_t tok = (static_cast<size_t>(b) * p.T + p.t_begin) * p.H + h;
            for (int i = tid; i < DK / 4; i += G::NT) {
                hd_cp16(S.k + 4 * i, p.k + tok * DK + 4 * i);
                hd_cp16(S.q + 4 * i, p.q + tok * DK + 4 * i);
            }
            for (int i = tid; i < DV / 4; i += G::NT) hd_cp16(S.v + 4 * i, p.v + tok * DV + 4 * i);
        }
    }
    hd_commit();
}

template <int DK, int DV>
__global__ void __launch_bounds__(HeadGeom<DK, DV>::NT, 2) head_wb_kernel(const StepParams p, int nheads) {
    using G = HeadGeom<DK, DV>;
    static_assert(G::ok, "head-unit layout");
    constexpr int NB = G::NB, NCS = G::NCS, CS = G::CS, CPL = G::CPL, NSG = G::NSG, NT = G::NT;
    using V = typename HeadLane<CPL>::V;
    using Sm = HeadSmem<DK, DV>;
    using St = HeadStage<DK, DV>;
    extern __shared__ __align__(16) uint8_t smem_raw[];
    Sm& sm = *reinterpret_cast<Sm*>(smem_raw);
    St* stg = reinterpret_cast<St*>(smem_raw + ((sizeof(Sm) + 15) & ~static_cast<size_t>(15)));
    const int pstride = (p.stage_bytes + 16 + 15) & ~15;
    uint8_t* pin0 = reinterpret_cast<uint8_t*>(stg + 2);
    uint8_t* pout = pin0 + 2 * pstride;
    __shared__ HeadMeta nmeta;   // the metadata of the head after the next

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int blk = warp / NCS, cs = warp - blk * NCS;
    const int r0 = 32 * blk;
    const int col0 = cs * CS + lane * CPL;
    const int soff = blk * DV + col0;   // the lane's first scale group within the head
    const bool has_tokens = p.t_end > p.t_begin;
    const bool stats = has_tokens && p.ema_s != nullptr;
    using Vec = typename std::conditional<DV == 128, uint4, uint2>::type;

    if (tid < kNFit) sm.fitf[tid] = fit_factor(tid);
    const int g_begin = static_cast<int>(static_cast<long long>(blockIdx.x) * nheads / gridDim.x);
    const int g_end = static_cast<int>(static_cast<long long>(blockIdx.x + 1) * nheads / gridDim.x);
    if (g_begin >= g_end) return;
    // the first head: metadata and copies; the second head's metadata
    auto scalars = [&](St& S, int bh, const HeadMeta& m) {   // one thread: first-token scalars
        const int b = bh / p.H, h = bh - b * p.H;
        const size_t tok = (static_cast<size_t>(b) * p.T + p.t_begin) * p.H + h;
        S.w_in = m.w_in; S.w_out = m.w_out; S.in_off = m.in_off; S.out_off = m.out_off; S.ok = m.ok;
        S.beta = (has_tokens && p.erase) ? __ldg(p.beta + tok) : 1.0f;
        S.rate = !has_tokens ? 1.0f
                 : p.s_code ? __ldg(p.s_lut + static_cast<size_t>(h) * p.L + min(static_cast<int>(p.s_code[tok]), p.L - 1))
                            : __ldg(p.s + tok);
        S.ms = stats ? __ldg(p.ema_s + bh) : 0.0f;
        S.mr = stats ? __ldg(p.ema_r + bh) : 0.0f;
    };
    {
        const HeadMeta m0 = head_meta<DK, DV>(p, g_begin);
        head_issue<DK, DV>(stg[0], pin0, m0, g_begin, p);
        if (tid == 0) {
            scalars(stg[0], g_begin, m0);
            if (g_begin + 1 < g_end) nmeta = head_meta<DK, DV>(p, g_begin + 1);
        }
    }
    float nbeta = 1.0f, nrate = 1.0f, nms = 0.0f, nmr = 0.0f;   // thread 0: next head's scalars
    HeadMeta m2;                                                   // thread 0: metadata two ahead
    m2.ok = 0;

    for (int bh = g_begin, j = 0; bh < g_end; ++bh, ++j) {
        St& S = stg[j & 1];
        uint8_t* pay = pin0 + (j & 1) * pstride;
        hd_wait_all();
        __syncthreads();                     // head bh's copies have landed; head bh - 1 is done
        const bool has_next = bh + 1 < g_end;
        if (has_next) {
            const HeadMeta mn = nmeta;
            head_issue<DK, DV>(stg[(j + 1) & 1], pin0 + ((j + 1) & 1) * pstride, mn, bh + 1, p);
            if (tid == 0) {
                // the next head's scalars and the metadata after it: loads now, stored below
                const int nb = (bh + 1) / p.H, nh = (bh + 1) - nb * p.H;
                const size_t ntok = (static_cast<size_t>(nb) * p.T + p.t_begin) * p.H + nh;
                nbeta = (has_tokens && p.erase) ? __ldg(p.beta + ntok) : 1.0f;
                nrate = !has_tokens ? 1.0f
                        : p.s_code ? __ldg(p.s_lut + static_cast<size_t>(nh) * p.L + min(static_cast<int>(p.s_code[ntok]), p.L - 1))
                                   : __ldg(p.s + ntok);
                nms = stats ? __ldg(p.ema_s + bh + 1) : 0.0f;
                nmr = stats ? __ldg(p.ema_r + bh + 1) : 0.0f;
                if (bh + 2 < g_end) m2 = head_meta<DK, DV>(p, bh + 2);
            }
        }
        const int b = bh / p.H, h = bh - b * p.H;
        if (!S.ok) {   // uniform: nothing of this head is touched
            if (tid == 0) raise_status(p.status, QS_DEV_LAYOUT);
            __syncthreads();
            if (tid == 0 && has_next) {
                St& N = stg[(j + 1) & 1];
                N.w_in = nmeta.w_in; N.w_out = nmeta.w_out; N.in_off = nmeta.in_off; N.out_off = nmeta.out_off;
                N.ok = nmeta.ok; N.beta = nbeta; N.rate = nrate; N.ms = nms; N.mr = nmr;
                nmeta = m2;
            }
            continue;
        }
        const int w_in = S.w_in, w_out = S.w_out;
        const int bytes_out = DK * DV / 8 * w_out;
        if (tid < 4) reinterpret_cast<uint32_t*>(pay + DK * DV / 8 * w_in)[tid] = 0u;   // readable tail
        // zero the output rows: codes are OR-ed in
        {
            const int nz = (bytes_out + 16) / 16;
            for (int i = tid; i < nz; i += NT) reinterpret_cast<uint4*>(pout)[i] = make_uint4(0, 0, 0, 0);
        }
        __syncthreads();                     // tail word written; stage scalars visible

        // ---- unpack + dequantise ------------------------------------------------------------------
        V x[32];
        {
            const float nA = -(8388608.0f + (w_in >= 2 ? static_cast<float>((1 << (w_in - 1)) - 1) : 0.0f));
            V S2, B2;
#pragma unroll
            for (int c = 0; c < CPL; ++c) {
                const float D = f16_value(S.sc[soff + c]);
                hv_set(S2, c, w_in >= 2 ? D : (w_in == 1 ? -2.0f * D : 0.0f));
                hv_set(B2, c, w_in == 1 ? D : 0.0f);
            }
            const V A2 = hv_bc<V>(nA);
            switch (w_in) {   // widths above 16 were rejected with the head's layout
#define QS_HU(N) case N: head_unpack_rows<N, DV, CPL, V>(pay, r0, col0, A2, S2, B2, x); break;
                QS_HU(0) QS_HU(1) QS_HU(2) QS_HU(3) QS_HU(4) QS_HU(5) QS_HU(6) QS_HU(7) QS_HU(8)
                QS_HU(9) QS_HU(10) QS_HU(11) QS_HU(12) QS_HU(13) QS_HU(14) QS_HU(15) QS_HU(16)
#undef QS_HU
                default:
#pragma unroll
                    for (int r = 0; r < 32; ++r) x[r] = hv_bc<V>(0.0f);
            }
        }

        // ---- tokens (Eq. 1) ----------------------------------------------------------------------
        if (stats && tid == DV) {
            sm.ms = S.ms;
            sm.mr = S.mr;
        }
        for (int t = p.t_begin; t < p.t_end; ++t) {
            const bool first = t == p.t_begin;
            if (!first) __syncthreads();     // every warp is done with the previous token's k, u
            const size_t tok = (static_cast<size_t>(b) * p.T + t) * p.H + h;
            const float beta = first ? S.beta : (p.erase ? __ldg(p.beta + tok) : 1.0f);
            const float rate = first ? S.rate
                                     : p.s_code ? __ldg(p.s_lut + static_cast<size_t>(h) * p.L +
                                                        min(static_cast<int>(p.s_code[tok]), p.L - 1))
                                                : __ldg(p.s + tok);
            if (tid == 0 && (!(rate > 0.0f) || !(rate < INFINITY))) raise_status(p.status, QS_DEV_RATE);
            if (tid < DK) {
                const int i = tid;
                const float kk = first ? S.k[i] : __ldg(p.k + tok * DK + i);
                const float qq = first ? S.q[i] : __ldg(p.q + tok * DK + i);
                const float ai = p.general ? __ldg(p.a_in + tok * DK + i) : __fmul_rn(beta, kk);
                sm.aq[i] = make_float4(ai, ai, qq, qq);
                sm.kk[i] = make_float2(kk, kk);
                const float kq = warp_sum(kk * qq);
                const float k2 = warp_sum(kk * kk);
                float ak = 0.0f, aa = 0.0f;
                if (p.general) {
                    ak = warp_sum(ai * kk);
                    aa = warp_sum(ai * ai);
                }
                if (lane == 0) {
                    sm.wsum[0][warp] = kq;
                    sm.wsum[1][warp] = k2;
                    sm.wsum[2][warp] = ak;
                    sm.wsum[3][warp] = aa;
                }
            }
            if (tid < DV) {
                sm.v[tid] = first ? S.v[tid] : __ldg(p.v + tok * DV + tid);
                if (p.general) sm.gw[tid] = __ldg(p.w_in + tok * DV + tid);
            }
            __syncthreads();
            const V d2 = hv_bc<V>(expf(-rate));
            V pp = hv_bc<V>(0.0f), rr = hv_bc<V>(0.0f);
#pragma unroll
            for (int r = 0; r < 32; ++r) {
                const float4 aq = sm.aq[r0 + r];
                x[r] = hv_mul(x[r], d2);
                if constexpr (CPL == 2) {
                    pp = hv_fma(x[r], make_float2(aq.x, aq.y), pp);
                    rr = hv_fma(x[r], make_float2(aq.z, aq.w), rr);
                } else {
                    pp = hv_fma(x[r], aq.x, pp);
                    rr = hv_fma(x[r], aq.z, rr);
                }
            }
#pragma unroll
            for (int c = 0; c < CPL; ++c) {
                sm.red[0][blk][col0 + c] = hv_get(pp, c);
                sm.red[1][blk][col0 + c] = hv_get(rr, c);
            }
            __syncthreads();
            if (tid < DV) {
                const int jv = tid;
                float Pp = 0.0f, Rr = 0.0f, kq = 0.0f;
#pragma unroll
                for (int k = 0; k < NB; ++k) {
                    Pp += sm.red[0][k][jv];
                    Rr += sm.red[1][k][jv];
                }
#pragma unroll
                for (int w = 0; w < DK / 32; ++w) kq += sm.wsum[0][w];
                const float vj = sm.v[jv];
                const float wj = p.general ? sm.gw[jv] : beta;
                const float u = (p.erase || p.general) ? __fsub_rn(__fmul_rn(wj, vj), Pp) : vj;
                sm.u[jv] = u;
                p.o[tok * DV + jv] = fmaf(u, kq, Rr);
            }
            if (stats && tid == DV) {   // Sec. 3 statistics per head (a thread with no column)
                float k2 = 0.0f;
#pragma unroll
                for (int w = 0; w < DK / 32; ++w) k2 += sm.wsum[1][w];
                const float xs = -expm1f(-2.0f * rate);
                float xr = p.erase ? __fmul_rn(__fmul_rn(beta, __fsub_rn(2.0f, beta)),
                                               __fdiv_rn(k2, static_cast<float>(DK)))
                                   : 0.0f;
                if (p.general) {
                    float ak = 0.0f, aa = 0.0f;
#pragma unroll
                    for (int w = 0; w < DK / 32; ++w) {
                        ak += sm.wsum[2][w];
                        aa += sm.wsum[3][w];
                    }
                    xr = __fdiv_rn(__fsub_rn(__fmul_rn(2.0f, ak), __fmul_rn(aa, k2)), static_cast<float>(DK));
                }
                if (t == 0) {
                    sm.ms = xs;
                    sm.mr = xr;
                } else {
                    sm.ms = __fadd_rn(sm.ms, __fmul_rn(p.alpha, __fsub_rn(xs, sm.ms)));
                    sm.mr = __fadd_rn(sm.mr, __fmul_rn(p.alpha, __fsub_rn(xr, sm.mr)));
                }
            }
            __syncthreads();
            V u2;
#pragma unroll
            for (int c = 0; c < CPL; ++c) hv_set(u2, c, sm.u[col0 + c]);
#pragma unroll
            for (int r = 0; r < 32; ++r) {
                if constexpr (CPL == 2) x[r] = hv_fma(sm.kk[r0 + r], u2, x[r]);
                else x[r] = hv_fma(sm.kk[r0 + r].x, u2, x[r]);
            }
        }
        // the next head's scalars (their loads were issued at this head's start)
        if (tid == 0 && has_next) {
            St& N = stg[(j + 1) & 1];
            N.w_in = nmeta.w_in; N.w_out = nmeta.w_out; N.in_off = nmeta.in_off; N.out_off = nmeta.out_off;
            N.ok = nmeta.ok; N.beta = nbeta; N.rate = nrate; N.ms = nms; N.mr = nmr;
            nmeta = m2;
        }

        // ---- write-back ---------------------------------------------------------------------------
        {
            const int w = w_out;
            const bool refit = (p.fit_every <= 1) || ((p.w_index + h) % p.fit_every == 0);
            V Rg = hv_bc<V>(0.0f), Mg = hv_bc<V>(0.0f);
#pragma unroll
            for (int r = 0; r < 32; ++r) {
#pragma unroll
                for (int c = 0; c < CPL; ++c) {
                    const float av = fabsf(hv_get(x[r], c));
                    hv_set(Rg, c, fmaxf(hv_get(Rg, c), av));
                    if (w == 1) hv_set(Mg, c, __fadd_rn(hv_get(Mg, c), av));   // in row order
                }
            }
            int fidx[CPL];
            float D[CPL];
            const float nf = w >= 2 ? static_cast<float>((1 << (w - 1)) - 1) : 0.0f;
            const float inv_n = w >= 2 ? __frcp_rn(nf) : 0.0f;
#pragma unroll
            for (int c = 0; c < CPL; ++c) {
                fidx[c] = static_cast<int>(S.fidx[soff + c]);
                D[c] = 0.0f;
            }
            if (w == 1) {
#pragma unroll
                for (int c = 0; c < CPL; ++c) D[c] = f16_round(__fdiv_rn(hv_get(Mg, c), 32.0f));
            } else if (w >= 2 && refit) {
                // From f = 1 down, one candidate per round; the clipping error of the group's
                // maximum bounds a candidate's error from below and grows as f falls, so once it
                // exceeds the best error found (2^-10 margin) the search stops (exact).  Equal
                // errors go to the larger factor.  Approximate reciprocals in the search; the
                // chosen step's IEEE reciprocal for the codes.
                float best[CPL];
#pragma unroll
                for (int c = 0; c < CPL; ++c) {
                    best[c] = INFINITY;
                    fidx[c] = kNFit - 1;
                }
                const float lim = kMagic + nf;
                const V M2 = hv_bc<V>(kMagic), nM2 = hv_bc<V>(-kMagic);
#pragma unroll 1
                for (int k = kNFit - 1; k >= 0; --k) {
                    const float f = sm.fitf[k];
                    V iv, nd;
                    bool go[CPL], any = false;
#pragma unroll
                    for (int c = 0; c < CPL; ++c) {
                        const float R = hv_get(Rg, c);
                        const float Dk = R > 0.0f ? cand_step(f, R, inv_n) : 0.0f;
                        float ik = 0.0f;
                        if (Dk > 0.0f) asm("rcp.approx.ftz.f32 %0, %1;" : "=f"(ik) : "f"(Dk));
                        hv_set(iv, c, ik);
                        hv_set(nd, c, -Dk);
                        const float e = fmaxf(R - nf * Dk, 0.0f);
                        go[c] = R > 0.0f && e * e <= best[c] * (1.0f + 1.0f / 1024.0f);
                        any |= go[c];
                    }
                    if (!__any_sync(kFull, any)) break;
                    V a0 = hv_bc<V>(0.0f), a1 = hv_bc<V>(0.0f);
#pragma unroll
                    for (int r = 0; r < 32; r += 2) {
                        V t0 = hv_fma(hv_abs(x[r]), iv, M2), t1 = hv_fma(hv_abs(x[r + 1]), iv, M2);
#pragma unroll
                        for (int c = 0; c < CPL; ++c) {
                            hv_set(t0, c, fminf(hv_get(t0, c), lim));
                            hv_set(t1, c, fminf(hv_get(t1, c), lim));
                        }
                        const V e0 = hv_fma(hv_add(t0, nM2), nd, hv_abs(x[r]));
                        const V e1 = hv_fma(hv_add(t1, nM2), nd, hv_abs(x[r + 1]));
                        a0 = hv_fma(e0, e0, a0);
                        a1 = hv_fma(e1, e1, a1);
                    }
                    const V acc = hv_add(a0, a1);
#pragma unroll
                    for (int c = 0; c < CPL; ++c) {
                        if (go[c] && hv_get(acc, c) < best[c]) {
                            best[c] = hv_get(acc, c);
                            fidx[c] = k;
                        }
                    }
                }
#pragma unroll
                for (int c = 0; c < CPL; ++c) {
                    const float R = hv_get(Rg, c);
                    if (R == 0.0f) fidx[c] = kNFit - 1;
                    D[c] = R > 0.0f ? cand_step(sm.fitf[fidx[c]], R, inv_n) : 0.0f;
                }
            } else if (w >= 2) {
#pragma unroll
                for (int c = 0; c < CPL; ++c) {
                    const float R = hv_get(Rg, c);
                    D[c] = R > 0.0f ? cand_step(sm.fitf[fidx[c]], R, inv_n) : 0.0f;
                }
            }
            if (w >= 1) {
                V inv2;
#pragma unroll
                for (int c = 0; c < CPL; ++c) hv_set(inv2, c, step_rcp(D[c]));
                switch (w) {
#define QS_HP(N) case N: head_pack_rows<N, DV, CPL, V>(x, inv2, pout, r0, col0); break;
                    QS_HP(1) QS_HP(2) QS_HP(3) QS_HP(4) QS_HP(5) QS_HP(6) QS_HP(7) QS_HP(8)
                    QS_HP(9) QS_HP(10) QS_HP(11) QS_HP(12) QS_HP(13) QS_HP(14) QS_HP(15) QS_HP(16)
#undef QS_HP
                    default: break;
                }
            }
            const size_t gb = static_cast<size_t>(bh) * NSG + soff;
#pragma unroll
            for (int c = 0; c < CPL; ++c) {
                p.out_scales[gb + c] = f16_bits(D[c]);
                p.out_fidx[gb + c] = static_cast<uint8_t>(fidx[c]);
            }
            __syncthreads();
            Vec* dst = reinterpret_cast<Vec*>(p.out_payload + static_cast<size_t>(b) * p.region_bytes + S.out_off);
            const Vec* srcv = reinterpret_cast<const Vec*>(pout);
            for (int i = tid; i < bytes_out / static_cast<int>(sizeof(Vec)); i += NT) dst[i] = srcv[i];
        }
        if (stats && tid == DV) {
            p.ema_s[bh] = sm.ms;
            p.ema_r[bh] = sm.mr;
        }
    }
}

template <int DK, int DV>
size_t head_wb_smem(int stage_bytes) {
    const size_t pstride = (static_cast<size_t>(stage_bytes) + 16 + 15) & ~static_cast<size_t>(15);
    return ((sizeof(HeadSmem<DK, DV>) + 15) & ~static_cast<size_t>(15)) + 2 * sizeof(HeadStage<DK, DV>) + 3 * pstride;
}

template <int DK, int DV>
cudaError_t launch_head_wb_t(const qstate_cfg& cfg, const StepParams& p, cudaStream_t stream) {
    auto kern = head_wb_kernel<DK, DV>;
    StepParams q = p;
    q.stage_bytes = DK * DV * cfg.bmax / 8;
    const size_t smem = head_wb_smem<DK, DV>(q.stage_bytes);
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
    if (e != cudaSuccess) return e;
    int dev = 0, sms = 0, per_sm = 0;
    if ((e = cudaGetDevice(&dev)) != cudaSuccess) return e;
    if ((e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess) return e;
    if ((e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, HeadGeom<DK, DV>::NT, smem)) != cudaSuccess) return e;
    const int nheads = cfg.B * cfg.H;
    const int grid = std::min(nheads, std::max(1, per_sm) * sms);
    kern<<<grid, HeadGeom<DK, DV>::NT, smem, stream>>>(q, nheads);
    return cudaGetLastError();
}

}  // namespace qs
