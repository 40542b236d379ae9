// qs_step_impl.cuh -- general write-back kernel of libqstate for the row allocation unit (sm_103a);
// the head unit has its own kernel (qs_head.cuh).
//
// One CTA per (batch element, head), 8 warps.  Warp w owns key rows [w*RPW, (w+1)*RPW); lane
// l owns value columns [l*CPL, (l+1)*CPL) of each of them, so one row is handled by one warp
// and its bit width is warp-uniform.  The head's FP32 state lives in registers for the whole
// write-back interval:
//   1. metadata: widths -> row byte offsets by prefix sums (Sec. 3, "Prefix sums of widths give
//      row offsets"), layout check, per-row dequantisation constants, shared tables;
//   2. the head's packed rows are staged in shared memory with 16-byte (dv = 128) or 8-byte
//      (dv = 64) vector loads;
//   3. unpack + dequantise (Sec. 3 levels), branch-free: x = (float(u) - A) S + Bc per row;
//   4. per token (Eq. 1): decay, fused reductions p = (beta k)^T S', r = q^T S' (per-lane
//      partials over the warp's rows, then across warps in shared memory), delta update,
//      readout o = S^T q = r + u (k . q) before quantisation (Sec. 2), EMA statistics (Sec. 3);
//   5. write-back (Sec. 3, "Levels and storage"): row ranges by warp reductions; the scalar
//      per-row work (16 candidate FP16 steps and their reciprocals) row-parallel, one thread
//      per row, into a shared table; then per row the squared-error search over the candidates,
//      codes, and the row's bits OR-ed into a zeroed shared staging row; finally one vector
//      store of the head's new region and coalesced stores of scales / factors / ranges.
// The same template serves pack (dense -> packed, no tokens), unpack (packed -> dense) and the
// unquantised reference path (dense -> dense).
#pragma once

#include <type_traits>

#include "qs_common.cuh"
#include "qs_head.cuh"

namespace qs {

template <int DK, int DV>
struct alignas(16) StepSmem {
    static constexpr int NW = 8;
    static constexpr int NSG = DK;
    float cand[DK][kNFit][2];             // (Delta_k, 1/Delta_k) of the refit rows
    float k[DK], q[DK], d[DK];
    float v[DV], u[DV];
    float ga[DK], gw[DV];                 // general erasure: this token's a and w
    float red[2][NW][DV];                 // p and r partials per warp
    float scale_in[NSG];                  // source steps / means (float)
    float ms[DK], mr[DK];                 // EMA statistics per row
    float deqA[DK], deqS[DK], deqB[DK];   // row unit dequantisation constants
    float rowR[DK], rowM[DK], rowD[DK], rowInv[DK];
    float fitf[kNFit];                    // f_k = (5 + k) / 20
    float inv_n[17];                      // 1 / (2^(w-1) - 1), w = 2..16
    float wsum[4][NW];                    // per-warp partial k.q, |k|^2, a.k, |a|^2
    int off_in[DK + 1], off_out[DK + 1];  // row byte offsets inside the head (+ total)
    uint16_t out_scale[NSG];
    uint8_t out_fidx[NSG];
    uint8_t w_in[DK], w_out[DK];
    uint8_t fidx_in[NSG];
    uint8_t mode[DK];                     // row unit: 1 = search the 16 candidates
    int flag;
};

// Sum 16 per-lane values over the warp by recursive halving; lane l ends with the total of
// value index (l >> 1) & 15.
__device__ __forceinline__ float reduce16(float (&v)[16], int lane) {
#pragma unroll
    for (int st = 0; st < 4; ++st) {
        const int half = 8 >> st;
        const int off = 16 >> st;
        const bool upper = (lane & off) != 0;
#pragma unroll
        for (int i = 0; i < half; ++i) {
            float send = upper ? v[i] : v[i + half];
            float keep = upper ? v[i + half] : v[i];
            v[i] = keep + __shfl_xor_sync(kFull, send, off);
        }
    }
    return v[0] + __shfl_xor_sync(kFull, v[0], 1);
}

// OR a lane's CPL codes (w bits each, CPL*w <= 64) into a zeroed shared row at bit
// lane*CPL*w.  `words` is the row's first 32-bit word.
template <int CPL>
__device__ __forceinline__ void or_codes(uint32_t* words, int lane, int w, const uint32_t (&u)[CPL]) {
    uint64_t chunk = 0;
#pragma unroll
    for (int c = 0; c < CPL; ++c) chunk |= static_cast<uint64_t>(u[c]) << (c * w);
    const int P = lane * CPL * w;
    const int idx = P >> 5, sh = P & 31;
    const uint64_t lo = chunk << sh;
    const uint32_t hi = sh ? static_cast<uint32_t>(chunk >> (64 - sh)) : 0u;
    const uint32_t w0 = static_cast<uint32_t>(lo), w1 = static_cast<uint32_t>(lo >> 32);
    if (w0) atomicOr(words + idx, w0);
    if (w1) atomicOr(words + idx + 1, w1);
    if (hi) atomicOr(words + idx + 2, hi);
}

template <int DK, int DV, bool SRC_PACKED, bool DST_PACKED>
__global__ void __launch_bounds__(256, 2) step_kernel(const StepParams p) {
    constexpr int NW = 8, RPW = DK / NW, CPL = DV / 32;
    using Sm = StepSmem<DK, DV>;
    constexpr int NSG = Sm::NSG;
    extern __shared__ __align__(16) uint8_t smem_raw[];
    Sm& sm = *reinterpret_cast<Sm*>(smem_raw);
    uint8_t* pay = smem_raw + sizeof(Sm);

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int bh = blockIdx.x, b = bh / p.H, h = bh - b * p.H;
    const size_t ubase = static_cast<size_t>(bh) * DK;
    const size_t gbase = static_cast<size_t>(bh) * NSG;
    const bool has_tokens = p.t_end > p.t_begin;
    const bool stats = has_tokens && p.ema_s != nullptr;

    // ---- 1. metadata ---------------------------------------------------------------------
    if (tid == 0) sm.flag = 0;
    if (tid < kNFit) sm.fitf[tid] = fit_factor(tid);
    if (tid >= 32 && tid < 32 + 17) {
        const int w = tid - 32;
        sm.inv_n[w] = w >= 2 ? __frcp_rn(static_cast<float>((1 << (w - 1)) - 1)) : 0.0f;
    }
    if (SRC_PACKED) {
        for (int i = tid; i < DK; i += 256) sm.w_in[i] = p.in_widths[ubase + i];
        for (int g = tid; g < NSG; g += 256) sm.scale_in[g] = f16_value(p.in_scales[gbase + g]);
    }
    if (DST_PACKED) {
        for (int i = tid; i < DK; i += 256) sm.w_out[i] = p.out_widths[ubase + i];
        for (int g = tid; g < NSG; g += 256) sm.fidx_in[g] = p.in_fidx ? p.in_fidx[gbase + g] : 15;
    }
    if (stats) {
        for (int i = tid; i < DK; i += 256) {
            sm.ms[i] = p.ema_s[ubase + i];
            sm.mr[i] = p.ema_r[ubase + i];
        }
    }
    __syncthreads();
    if ((warp == 0 && SRC_PACKED) || (warp == 1 && DST_PACKED)) {
        const uint8_t* wa = warp == 0 ? sm.w_in : sm.w_out;
        int* off = warp == 0 ? sm.off_in : sm.off_out;
        constexpr int PER = DK / 32;
        int loc[PER];
        int sum = 0;
        bool bad = false;
#pragma unroll
        for (int j = 0; j < PER; ++j) {
            const int w = wa[lane * PER + j];
            bad |= (w > 16);
            loc[j] = sum;
            sum += w * (DV / 8);
        }
        int incl = sum;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int n = __shfl_up_sync(kFull, incl, o);
            if (lane >= o) incl += n;
        }
        const int excl = incl - sum;
#pragma unroll
        for (int j = 0; j < PER; ++j) off[lane * PER + j] = excl + loc[j];
        const int total = __shfl_sync(kFull, incl, 31);
        bad = __any_sync(kFull, bad);
        const long long hoff = warp == 0 ? p.in_head_off[bh] : p.out_head_off[bh];
        const int align = (DV == 128) ? 16 : 8;
        if (lane == 0) {
            off[DK] = total;
            if (bad || hoff + total > p.region_bytes || (hoff % align) != 0 || total > p.stage_bytes)
                atomicExch(&sm.flag, 1);
        }
    }
    if (SRC_PACKED && tid >= 64 && tid < 64 + DK) {
        // per-row dequantisation x = (float(u) - A) S + Bc: w >= 2 -> (q) Delta; w = 1 -> +-m;
        // w = 0 -> 0 (float(u) is 2^23 + u built from the code bits)
        const int i = tid - 64;
        const int w = min(static_cast<int>(sm.w_in[i]), 16);
        const float D = sm.scale_in[i];
        sm.deqA[i] = 8388608.0f + static_cast<float>(w >= 2 ? (1 << (w - 1)) - 1 : 0);
        sm.deqS[i] = w >= 2 ? D : (w == 1 ? -2.0f * D : 0.0f);
        sm.deqB[i] = w == 1 ? D : 0.0f;
    }
    __syncthreads();
    if (sm.flag) {
        if (tid == 0) raise_status(p.status, QS_DEV_LAYOUT);
        return;
    }

    // ---- 2. stage the source rows in shared memory ----------------------------------------
    using Vec = typename std::conditional<DV == 128, uint4, uint2>::type;
    if (SRC_PACKED) {
        const int nbytes = sm.off_in[DK];
        const Vec* src = reinterpret_cast<const Vec*>(
            p.in_payload + static_cast<size_t>(b) * p.region_bytes + p.in_head_off[bh]);
        Vec* dst = reinterpret_cast<Vec*>(pay);
        const int nv = nbytes / static_cast<int>(sizeof(Vec));
        for (int i = tid; i < nv; i += 256) dst[i] = __ldg(src + i);
        if (tid < 4) reinterpret_cast<uint32_t*>(pay + nbytes)[tid] = 0u;
        __syncthreads();
    }

    // ---- 3. unpack + dequantise into registers ---------------------------------------------
    float x[RPW][CPL];
#pragma unroll
    for (int r = 0; r < RPW; ++r) {
        const int i = warp * RPW + r;
        if (SRC_PACKED) {
            const int w = sm.w_in[i];
            uint32_t u[CPL];
            extract_codes<CPL>(pay + sm.off_in[i], lane, w, u);
            const float A = sm.deqA[i], S = sm.deqS[i], Bc = sm.deqB[i];
#pragma unroll
            for (int c = 0; c < CPL; ++c)
                x[r][c] = fmaf(__fsub_rn(__uint_as_float(kTwo23Bits | u[c]), A), S, Bc);
        } else if (p.dense_in != nullptr) {
            const float* src = p.dense_in + (static_cast<size_t>(bh) * DK + i) * DV + lane * CPL;
            if (CPL == 4) {
                const float4 t = *reinterpret_cast<const float4*>(src);
                x[r][0] = t.x; x[r][1] = t.y; x[r][CPL > 2 ? 2 : 0] = t.z; x[r][CPL > 3 ? 3 : 0] = t.w;
            } else {
                const float2 t = *reinterpret_cast<const float2*>(src);
                x[r][0] = t.x; x[r][1] = t.y;
            }
        } else {
#pragma unroll
            for (int c = 0; c < CPL; ++c) x[r][c] = 0.0f;
        }
    }
    if (SRC_PACKED) __syncthreads();   // the staging buffer is reused for the output rows
    if (DST_PACKED) {                  // zero the output rows: codes are OR-ed in
        const int nz = (sm.off_out[DK] + 16) / 16;
        for (int i = tid; i < nz; i += 256) reinterpret_cast<uint4*>(pay)[i] = make_uint4(0, 0, 0, 0);
        if (!has_tokens) __syncthreads();
    }

    // ---- 4. tokens of this write-back interval (Eq. 1) --------------------------------------
    for (int t = p.t_begin; t < p.t_end; ++t) {
        if (t > p.t_begin) __syncthreads();   // every warp is done with the previous token's k, u
        const size_t tok = (static_cast<size_t>(b) * p.T + t) * p.H + h;
        const float beta = p.erase ? __ldg(p.beta + tok) : 1.0f;
        float rate_h = 0.0f;
        if (!p.decay_row)
            rate_h = p.s_code ? __ldg(p.s_lut + static_cast<size_t>(h) * p.L +
                                      min(static_cast<int>(p.s_code[tok]), p.L - 1))
                              : __ldg(p.s + tok);
        if (tid < DK) {
            const int i = tid;
            const float kk = __ldg(p.k + tok * DK + i), qq = __ldg(p.q + tok * DK + i);
            sm.k[i] = kk;
            sm.q[i] = qq;
            float rate = rate_h;
            if (p.decay_row)
                rate = p.s_code ? __ldg(p.s_lut + (static_cast<size_t>(h) * DK + i) * p.L +
                                        min(static_cast<int>(p.s_code[tok * DK + i]), p.L - 1))
                                : __ldg(p.s + tok * DK + i);
            if (!(rate > 0.0f) || !(rate < INFINITY)) raise_status(p.status, QS_DEV_RATE);
            sm.d[i] = expf(-rate);
            const float ai = p.general ? __ldg(p.a_in + tok * DK + i) : __fmul_rn(beta, kk);
            sm.ga[i] = ai;
            // Sec. 3 statistics per row (general erasure: after the barrier, as the erasure
            // term needs all of k)
            if (stats && !p.general) {
                const float xs = -expm1f(-2.0f * rate);
                const float xr = p.erase ? __fmul_rn(__fmul_rn(beta, __fsub_rn(2.0f, beta)), __fmul_rn(kk, kk)) : 0.0f;
                if (t == 0) {
                    sm.ms[i] = xs;
                    sm.mr[i] = xr;
                } else {
                    sm.ms[i] = __fadd_rn(sm.ms[i], __fmul_rn(p.alpha, __fsub_rn(xs, sm.ms[i])));
                    sm.mr[i] = __fadd_rn(sm.mr[i], __fmul_rn(p.alpha, __fsub_rn(xr, sm.mr[i])));
                }
            }
            const float kq = warp_sum(kk * qq);
            const float k2 = warp_sum(kk * kk);
            const float ak = warp_sum(ai * kk);
            const float aa = warp_sum(ai * ai);
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
        if (stats && p.general && tid < DK) {   // Sec. 3 statistics per row
            const int i = tid;
            float rate = rate_h;
            if (p.decay_row)
                rate = p.s_code ? __ldg(p.s_lut + (static_cast<size_t>(h) * DK + i) * p.L +
                                        min(static_cast<int>(p.s_code[tok * DK + i]), p.L - 1))
                                : __ldg(p.s + tok * DK + i);
            const float xs = -expm1f(-2.0f * rate);
            const float xr = general_erasure<DK>(sm.ga[i], sm.k[i], sm.k);
            if (t == 0) {
                sm.ms[i] = xs;
                sm.mr[i] = xr;
            } else {
                sm.ms[i] = __fadd_rn(sm.ms[i], __fmul_rn(p.alpha, __fsub_rn(xs, sm.ms[i])));
                sm.mr[i] = __fadd_rn(sm.mr[i], __fmul_rn(p.alpha, __fsub_rn(xr, sm.mr[i])));
            }
        }

        // decay and per-lane partial reductions over the warp's rows
        float pp[CPL], rr[CPL];
#pragma unroll
        for (int c = 0; c < CPL; ++c) pp[c] = rr[c] = 0.0f;
#pragma unroll
        for (int r = 0; r < RPW; ++r) {
            const int i = warp * RPW + r;
            const float d = sm.d[i];
            const float a = sm.ga[i];   // erase vector: beta k (delta rule) or the given a
            const float qi = sm.q[i];
#pragma unroll
            for (int c = 0; c < CPL; ++c) {
                x[r][c] = __fmul_rn(x[r][c], d);
                pp[c] = fmaf(x[r][c], a, pp[c]);
                rr[c] = fmaf(x[r][c], qi, rr[c]);
            }
        }
#pragma unroll
        for (int c = 0; c < CPL; ++c) {
            sm.red[0][warp][lane * CPL + c] = pp[c];
            sm.red[1][warp][lane * CPL + c] = rr[c];
        }
        __syncthreads();
        if (tid < DV) {
            const int j = tid;
            float P = 0.0f, Rr = 0.0f, kq = 0.0f;
#pragma unroll
            for (int w = 0; w < NW; ++w) {
                P += sm.red[0][w][j];
                Rr += sm.red[1][w][j];
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
        __syncthreads();
#pragma unroll
        for (int r = 0; r < RPW; ++r) {
            const float ki = sm.k[warp * RPW + r];
#pragma unroll
            for (int c = 0; c < CPL; ++c) x[r][c] = fmaf(ki, sm.u[lane * CPL + c], x[r][c]);
        }
    }

    // ---- 5. write-back ------------------------------------------------------------------------
    if (DST_PACKED) {
        const bool refit = (p.fit_every <= 1) || ((p.w_index + h) % p.fit_every == 0);
        {
            // (a) row ranges (and 1-bit means) by warp reductions
#pragma unroll
            for (int r = 0; r < RPW; ++r) {
                const int i = warp * RPW + r;
                float amax = 0.0f, asum = 0.0f;
#pragma unroll
                for (int c = 0; c < CPL; ++c) {
                    amax = fmaxf(amax, fabsf(x[r][c]));
                    asum += fabsf(x[r][c]);
                }
                const float R = warp_absmax(amax);
                if (sm.w_out[i] == 1) asum = warp_sum(asum);
                if (lane == 0) {
                    sm.rowR[i] = R;
                    sm.rowM[i] = asum;
                }
            }
            __syncthreads();
            // (b) scalar per-row work, one thread per row
            if (tid < DK) {
                const int i = tid, w = sm.w_out[i];
                const float R = sm.rowR[i];
                float D = 0.0f, inv = 0.0f;
                int fidx = sm.fidx_in[i], mode = 0;
                if (w == 1) {
                    D = f16_round(__fdiv_rn(sm.rowM[i], static_cast<float>(DV)));
                } else if (w >= 2) {
                    const float inv_n = sm.inv_n[w];
                    if (R == 0.0f) {
                        if (refit) fidx = kNFit - 1;
                    } else if (refit) {
                        mode = 1;
#pragma unroll 4
                        for (int k = 0; k < kNFit; ++k) {
                            const float Dk = cand_step(sm.fitf[k], R, inv_n);
                            sm.cand[i][k][0] = Dk;
                            sm.cand[i][k][1] = step_rcp(Dk);
                        }
                    } else {
                        D = cand_step(sm.fitf[fidx], R, inv_n);
                        inv = step_rcp(D);
                    }
                }
                sm.rowD[i] = D;
                sm.rowInv[i] = inv;
                sm.mode[i] = static_cast<uint8_t>(mode);
                sm.out_fidx[i] = static_cast<uint8_t>(fidx);
            }
            __syncthreads();
            // (c) per row: factor search, codes, bits into the staging row
#pragma unroll
            for (int r = 0; r < RPW; ++r) {
                const int i = warp * RPW + r;
                const int w = sm.w_out[i];
                uint32_t u[CPL];
                if (w >= 2) {
                    const int n = (1 << (w - 1)) - 1;
                    const float nf = static_cast<float>(n);
                    float D = sm.rowD[i], inv = sm.rowInv[i];
                    if (sm.mode[i]) {
                        const float4* ct = reinterpret_cast<const float4*>(&sm.cand[i][0][0]);
                        float sse[16];
#pragma unroll
                        for (int kk = 0; kk < 8; ++kk) {
                            const float4 cd = ct[kk];
                            float a0 = 0.0f, a1 = 0.0f;
#pragma unroll
                            for (int c = 0; c < CPL; ++c) {
                                const float a = fabsf(x[r][c]);
                                const float t0 = fminf(__fadd_rn(__fmul_rn(a, cd.y), kMagic), kMagic + nf);
                                const float e0 = fmaf(-__fsub_rn(t0, kMagic), cd.x, a);
                                a0 = fmaf(e0, e0, a0);
                                const float t1 = fminf(__fadd_rn(__fmul_rn(a, cd.w), kMagic), kMagic + nf);
                                const float e1 = fmaf(-__fsub_rn(t1, kMagic), cd.z, a);
                                a1 = fmaf(e1, e1, a1);
                            }
                            sse[2 * kk] = a0;
                            sse[2 * kk + 1] = a1;
                        }
                        const float tot = reduce16(sse, lane);
                        const unsigned sb = __float_as_uint(tot);
                        const unsigned mn = __reduce_min_sync(kFull, sb);
                        const int best = static_cast<int>(
                                             __reduce_max_sync(kFull, sb == mn ? ((lane >> 1) & 15) + 1 : 0u)) - 1;
                        D = sm.cand[i][best][0];
                        inv = sm.cand[i][best][1];
                        if (lane == 0) sm.out_fidx[i] = static_cast<uint8_t>(best);
                    }
                    if (lane == 0) sm.out_scale[i] = f16_bits(D);
#pragma unroll
                    for (int c = 0; c < CPL; ++c) {
                        const float tq = code_magic(x[r][c], inv, kMagic - nf, kMagic + nf);
                        u[c] = __float_as_uint(tq) - (kMagicBits - static_cast<uint32_t>(n));
                    }
                } else {
                    if (lane == 0) sm.out_scale[i] = f16_bits(sm.rowD[i]);
#pragma unroll
                    for (int c = 0; c < CPL; ++c) u[c] = (w == 1 && x[r][c] < 0.0f) ? 1u : 0u;
                }
                or_codes<CPL>(reinterpret_cast<uint32_t*>(pay + sm.off_out[i]), lane, w, u);
            }
        }
        __syncthreads();
        const int nbytes = sm.off_out[DK];
        Vec* dst = reinterpret_cast<Vec*>(p.out_payload + static_cast<size_t>(b) * p.region_bytes +
                                          p.out_head_off[bh]);
        const Vec* srcv = reinterpret_cast<const Vec*>(pay);
        const int nv = nbytes / static_cast<int>(sizeof(Vec));
        for (int i = tid; i < nv; i += 256) dst[i] = srcv[i];
        for (int g = tid; g < NSG; g += 256) {
            p.out_scales[gbase + g] = sm.out_scale[g];
            p.out_fidx[gbase + g] = sm.out_fidx[g];
        }
        if (p.range != nullptr)
            for (int i = tid; i < DK; i += 256) p.range[ubase + i] = sm.rowR[i];
    } else if (p.dense_out != nullptr) {
#pragma unroll
        for (int r = 0; r < RPW; ++r) {
            const int i = warp * RPW + r;
            float* dst = p.dense_out + (static_cast<size_t>(bh) * DK + i) * DV + lane * CPL;
            if (CPL == 4) {
                *reinterpret_cast<float4*>(dst) =
                    make_float4(x[r][0], x[r][1], x[r][CPL > 2 ? 2 : 0], x[r][CPL > 3 ? 3 : 0]);
            } else {
                *reinterpret_cast<float2*>(dst) = make_float2(x[r][0], x[r][1]);
            }
        }
    }
    if (stats) {
        for (int i = tid; i < DK; i += 256) {
            p.ema_s[ubase + i] = sm.ms[i];
            p.ema_r[ubase + i] = sm.mr[i];
        }
    }
}

template <int DK, int DV, bool SRC_PACKED, bool DST_PACKED>
cudaError_t launch_step_t(const qstate_cfg& cfg, const StepParams& p, cudaStream_t stream) {
    auto kern = step_kernel<DK, DV, SRC_PACKED, DST_PACKED>;
    const size_t smem = sizeof(StepSmem<DK, DV>) +
                        ((SRC_PACKED || DST_PACKED) ? static_cast<size_t>(DK) * DV * cfg.bmax / 8 + 32 : 0);
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         static_cast<int>(smem));
    if (e != cudaSuccess) return e;
    StepParams q = p;
    q.stage_bytes = DK * DV * cfg.bmax / 8;
    kern<<<cfg.B * cfg.H, 256, smem, stream>>>(q);
    return cudaGetLastError();
}

template <int DK, int DV>
cudaError_t launch_step_shape(const qstate_cfg& cfg, int src_packed, int dst_packed,
                              const StepParams& p, cudaStream_t stream) {
    // the allocation unit only shapes packing: dense -> dense runs the row-unit instance
    const bool head = cfg.unit_kind == QSTATE_UNIT_HEAD && (src_packed || dst_packed);
    if (head) {   // head unit: the kernel whose lanes own whole scale groups
        if constexpr (HeadGeom<DK, DV>::ok) {
            // a write-back whose per-head arrays are 16-byte aligned: the persistent kernel,
            // which copies the next head's inputs with cp.async while a head computes
            auto a16 = [](const void* q) { return q == nullptr || (reinterpret_cast<uintptr_t>(q) & 15u) == 0; };
            if (src_packed && dst_packed && p.t_end > p.t_begin && p.in_fidx && a16(p.in_payload) &&
                a16(p.out_payload) && a16(p.in_scales) && a16(p.in_fidx) && a16(p.k) && a16(p.q) && a16(p.v))
                return launch_head_wb_t<DK, DV>(cfg, p, stream);
            if (src_packed && dst_packed) return launch_head_t<DK, DV, true, true>(cfg, p, stream);
            if (!src_packed && dst_packed) return launch_head_t<DK, DV, false, true>(cfg, p, stream);
            return launch_head_t<DK, DV, true, false>(cfg, p, stream);
        }
        return cudaErrorInvalidValue;
    }
#define QS_CASE(SP, DP)                                                                \
    if ((src_packed != 0) == SP && (dst_packed != 0) == DP)                            \
        return launch_step_t<DK, DV, SP, DP>(cfg, p, stream);
    QS_CASE(true, true)
    QS_CASE(false, true)
    QS_CASE(true, false)
    QS_CASE(false, false)
#undef QS_CASE
    return cudaErrorInvalidValue;
}

}  // namespace qs
