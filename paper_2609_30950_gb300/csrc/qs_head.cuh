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
