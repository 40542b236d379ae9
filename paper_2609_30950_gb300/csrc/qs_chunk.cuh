// qs_chunk.cuh -- one write-back interval of a head in chunked form on the tensor cores
// (tcgen05, sm_103a), dk = dv = 128: the row-unit write-back kernel's alternative to its
// token-by-token loop (Eq. 1) for C > 1.
//
// Within a block of L = 16 tokens starting from state S_b, let d_t = e^{-s_t} (per key row),
// Dc_t = d_0 ... d_t (decay from S_b to token t's decayed state S'_t), a_t = beta_t k_t (or 0
// without erasure) and w_t = beta_t (or 1).  Unrolling Eq. (1) over the block gives, with
// P(s, t) = Dc_t / Dc_s = d_{s+1} ... d_t the decay between tokens s < t:
//     p_t = S'_t^T a_t = S_b^T (a_t o Dc_t) + sum_{s<t} A_ts u_s,   A_ts = sum_i a_ti k_si P_i(s, t)
//     u_t = w_t v_t - p_t
//     o_t = S_t^T q_t  = S_b^T (q_t o Dc_t) + sum_{s<=t} M_ts u_s,  M_ts = sum_i q_ti k_si P_i(s, t)
//     S_e = Dc_{L-1} o S_b + sum_t (k_t o Dc_{L-1} / Dc_t) u_t^T.
// The products with S_b (32 columns of S_b^T [a o Dc; q o Dc]^T), the matrices A and M (one
// product (k / Dc) [a o Dc; q o Dc]^T) and the state update (a rank-16 product) run on the
// tensor cores; the triangular solve for u and the readouts run on the CUDA cores.  The FP32 state stays in tensor memory (TMEM) as S^T (lane = value column j,
// column = key row i) for the whole interval: the FP32 value S and its remainder lo = S - hi
// below the top 19 bits hi.  The tensor core truncates its FP32 inputs to TF32, so reading S
// as an operand gives exactly hi; the products use the 3xTF32 scheme hi*hi + hi*lo + lo*hi.
// The tensor core's FP32 accumulation truncates, so large and small terms are kept apart: the
// hi*hi and the correction products of S_b^T [..] and of A and M go to separate accumulators
// (summed with one rounding when read), and the block's
// update goes to a fresh accumulator that the CUDA cores add to the decayed state with one
// rounding, S_e = fma(hi + lo, Dc_{L-1}, update).
//
// A and M are factored as (a o Dc) . (k / Dc) over the rows: exact while every Dc of a block
// stays a normal FP32 number, i.e. while the decay rates of one row sum to less than about 87
// over 16 tokens; a block beyond that raises QS_DEV_CHUNK (the token-by-token kernel has no such
// limit).
//
// Roles per block (256 threads): thread (row i, half) prepares key row i for 8 of the block's
// 16 tokens (rates, decays, EMA statistics, operand tiles); warps 4-7 also stage the next
// block's inputs and own value columns (TMEM lane j) for the solve; the readouts are split
// over both halves by token; all threads combine and split the state.
// Included by qs_wb_row.cuh, whose state-buffer swizzle sb_off it uses.
#pragma once

#include "qs_common.cuh"
#include "qs_tc.cuh"

namespace qs {

// Defined in qs_wb_row.cuh: the state buffer's swizzle (float offset of 16-byte group G of
// row i) and the cp.async helpers.
template <int DV>
__device__ __forceinline__ int sb_off(int i, int G);
__device__ __forceinline__ void cp_async16(void* smem, const void* gmem);
__device__ __forceinline__ void cp_async4(void* smem, const void* gmem);
__device__ __forceinline__ void cp_async_commit();
__device__ __forceinline__ void cp_async_wait_all();

struct ChunkGeo {
    static constexpr int L = 16;    // tokens per block
    static constexpr int D = 128;   // dk = dv
    // TMEM columns: S^T (FP32, read by the products as its TF32 part hi) and lo, the block's update, the product with S_b (hi*hi part and
    // corrections), u^T hi / lo, the product (k / Dc) [a o Dc ; q o Dc]^T that gives A and M
    static constexpr uint32_t kHi = 0, kLo = 128, kUpd = 256, kDW = 384, kDWc = 416, kUHi = 448,
                              kULo = 464, kAM = 480;
    // The correction products of A and M (hi*lo + lo*hi) accumulate apart from hi*hi, in the
    // update's columns: those are free from the state combine of one block to the update
    // product of the next, and A and M are read out before that product is issued.
    static constexpr uint32_t kAMc = kUpd;
    static constexpr uint32_t kCols = 512;
    // Operand tiles (K-major core matrices, see qs_tc.cuh).  A K-chunk is padded by 16 bytes
    // where a warp writes one column of consecutive key rows, so the writes spread over all
    // banks.
    //  k / Dc: L rows x D (K = key row), K-chunks 272 bytes apart.  It is the A operand of an
    //          M = 64 product: rows 16..63 alias the following bytes (always inside the
    //          region, read but never used), their output lanes are ignored.
    static constexpr uint32_t kLboH = L * 16 + 16, kSboH = 128;
    //  [a o Dc ; q o Dc]: 2L rows x D, K-chunks 528 bytes apart
    static constexpr uint32_t kLboW = 2 * L * 16 + 16, kSboW = 128;
    //  (k o Dc_{L-1} / Dc)^T: D rows (key rows) x L (K = token)
    static constexpr uint32_t kLboU = (D / 8) * 128, kSboU = 128;
    static constexpr uint32_t kKh = (D / 4) * kLboH, kBw = (D / 4) * kLboW, kBu = (L / 4) * kLboU;
    static constexpr uint32_t oKhHi = 0, oKhLo = kKh, oBwHi = 2 * kKh, oBwLo = 2 * kKh + kBw;
    static constexpr uint32_t oBuHi = 2 * kKh + 2 * kBw, oBuLo = oBuHi + kBu;
    static constexpr uint32_t oAM = oBuLo + kBu;                  // A and M, L x L each
    static constexpr uint32_t oDall = oAM + 2 * L * L * 4;        // two buffers, by block parity
    static constexpr uint32_t oXch = oDall + 2 * D * 4;          // row preparation: the halves' exchange
    // mbarriers of the products with S_b and A / M (two arrivals) and of the update (one); the
    // TMEM address (byte 16), the abort word (byte 20) and the teardown's mbarrier (byte 24)
    static constexpr uint32_t oBar = oXch + 2 * D * 16;
    // one block's token inputs, staged by cp.async: k, q, rates (FP32 per row, per head, or
    // uint8 codes) and beta (three buffers by block index mod 3: block c's solve still reads
    // its beta while block c + 2's arrives)
    static constexpr uint32_t oStg = oBar + 32;
    static constexpr uint32_t sK = 0, sQ = L * D * 4, sS = 2 * L * D * 4, sB = 3 * L * D * 4;
    static constexpr uint32_t kBytes = oStg + sB + 3 * L * 4;
};
static_assert(ChunkGeo::oBwHi % 16 == 0 && ChunkGeo::oBuHi % 16 == 0 && ChunkGeo::oBar % 16 == 0 &&
              ChunkGeo::oStg % 16 == 0, "tile alignment");
// the aliased rows of the k / Dc operand (16 row groups of 128 bytes from each K-step's start)
// stay inside the two k / Dc tiles and the first [a o Dc ; q o Dc] tile
static_assert(ChunkGeo::oKhLo + (ChunkGeo::D / 8 - 1) * 2 * ChunkGeo::kLboH + ChunkGeo::kLboH + 16 * 128 <=
              ChunkGeo::oBwLo, "aliased operand rows");

__device__ __forceinline__ volatile uint32_t* chunk_abort_word(uint8_t* cb) {
    return reinterpret_cast<volatile uint32_t*>(cb + ChunkGeo::oBar + 20);
}

// Wait for phase `parity` of a product mbarrier.  Gives up after `limit` polls (the call's
// wait_polls: kDefaultWaitPolls unless a caller lowered it) and then sets the CTA's abort word;
// once that word is set every later wait of the CTA gives up at once, so a product that never
// completes costs one limit, not one per wait.  A limit of 0 gives up without polling.
__device__ __forceinline__ bool chunk_wait(uint64_t* bar, uint32_t parity, volatile uint32_t* abort, int limit) {
    if (*abort != 0u) return false;
    for (int it = 0; it < limit; ++it) {
        if (tc::mbar_try_wait(bar, parity)) return true;
        if ((it & 255) == 255 && *abort != 0u) return false;
    }
    *abort = 1u;
    return false;
}

// Once per CTA: all 512 TMEM columns (the kernel runs one CTA per SM in this form) and the
// mbarriers of the products.  Returns the TMEM base address.
__device__ __forceinline__ uint32_t chunk_setup(uint8_t* cb) {
    using G = ChunkGeo;
    const int tid = threadIdx.x;
    uint64_t* bar = reinterpret_cast<uint64_t*>(cb + G::oBar);
    uint32_t* ta = reinterpret_cast<uint32_t*>(cb + G::oBar + 16);
    if (tid < 32) {
        tc::tmem_alloc(ta, G::kCols);
        tc::tmem_relinquish();
    }
    if (tid == 32) {
        tc::mbar_init(bar, 2);       // products with S_b (thread 0) and for A / M (thread 32)
        tc::mbar_init(bar + 1, 1);   // the update
        tc::mbar_init(bar + 3, 2);   // teardown after a wait gave up: both issuers' products
        *chunk_abort_word(cb) = 0u;
        tc::mbar_fence_init();
    }
    tc::fence_before_sync();
    __syncthreads();
    tc::fence_after_sync();
    return *ta;
}

// Frees the TMEM columns.  If a wait gave up (the abort word, uniform after the barrier),
// products may still be in flight: both issuing threads commit to the teardown mbarrier and
// warp 0 waits for it, bounded by the default limit whatever the call's own limit, before the
// columns are freed.  If that wait gives up too, QS_DEV_TEARDOWN is raised: the columns are
// freed all the same (holding them would block the next CTA's allocation for good), and the
// host then treats the device as unusable.  Copies in flight are waited for too.
__device__ __forceinline__ void chunk_teardown(uint32_t tmem, uint8_t* cb, int* status) {
    const int tid = threadIdx.x;
    cp_async_wait_all();
    tc::fence_before_sync();
    __syncthreads();
    if (*chunk_abort_word(cb) != 0u) {
        uint64_t* bar = reinterpret_cast<uint64_t*>(cb + ChunkGeo::oBar) + 3;
        if (tid == 0 || tid == 32) tc::mma_commit(bar);
        if (tid < 32 && !tc::mbar_wait(bar, 0u, kDefaultWaitPolls) && tid == 0)
            raise_status(status, QS_DEV_TEARDOWN);
    }
    if (tid < 32) {
        tc::fence_after_sync();
        tc::tmem_dealloc(tmem, ChunkGeo::kCols);
    }
}

// The interval [p.t_begin, p.t_end) of head (b, h): the state arrives in sbuf (row-major,
// swizzled) and leaves there; readouts go to p.o, the EMA statistics of the rows to S.ms / S.mr.
// `phase` tracks the mbarriers' parities (uniform over the CTA).
template <class Stage>
__device__ __forceinline__ void chunk_interval(const StepParams& p, Stage& S, float* sbuf, uint8_t* cb,
                                               uint32_t tmem, uint32_t& phase, int b, int h, bool stats) {
    using G = ChunkGeo;
    constexpr int L = G::L, D = G::D;
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int sub = warp & 3, hf = warp >> 2;
    const int jl = 32 * sub + lane;   // the TMEM lane (value column) this thread addresses
    const int tt = tid - 128;         // index among the value-column threads (warps 4-7)
    const uint32_t tl = tmem + (static_cast<uint32_t>(32 * sub) << 16);
    uint64_t* bar = reinterpret_cast<uint64_t*>(cb + G::oBar);
    float* amA = reinterpret_cast<float*>(cb + G::oAM);
    float* amM = amA + L * L;
    float* dall = reinterpret_cast<float*>(cb + G::oDall);
    uint8_t* kh_hi = cb + G::oKhHi;
    uint8_t* kh_lo = cb + G::oKhLo;
    uint8_t* bw_hi = cb + G::oBwHi;
    uint8_t* bw_lo = cb + G::oBwLo;
    uint8_t* bu_hi = cb + G::oBuHi;
    uint8_t* bu_lo = cb + G::oBuLo;
    uint8_t* stg = cb + G::oStg;
    const float* sk = reinterpret_cast<const float*>(stg + G::sK);
    const float* sq = reinterpret_cast<const float*>(stg + G::sQ);
    const float* ss = reinterpret_cast<const float*>(stg + G::sS);
    const uint8_t* sc = stg + G::sS;
    const size_t tokb = static_cast<size_t>(b) * p.T;
    // `phase` carries both mbarriers' parities: bit 0 the first's, bit 1 the second's
    volatile uint32_t* abort = chunk_abort_word(cb);
    auto wait_mma = [&](int which) {
        if (!chunk_wait(bar + which, (phase >> which) & 1u, abort, p.wait_polls)) raise_status(p.status, QS_DEV_TIMEOUT);
        phase ^= 1u << which;
        tc::fence_after_sync();
    };
    // staging of the block at token tb by the value-column threads: k, q, the rates and beta
    auto issue_kqs = [&](int tb) {
        const int nb = min(L, p.t_end - tb);
        if (p.erase && tt < nb)
            cp_async4(stg + G::sB + (((tb - p.t_begin) / L) % 3) * L * 4 + tt * 4, p.beta + (tokb + tb + tt) * p.H + h);
        for (int c = tt; c < nb * (D / 4); c += 128) {
            const int tau = c / (D / 4), part = c % (D / 4);
            const size_t tok = (tokb + tb + tau) * p.H + h;
            cp_async16(stg + G::sK + tau * D * 4 + part * 16, p.k + tok * D + part * 4);
            cp_async16(stg + G::sQ + tau * D * 4 + part * 16, p.q + tok * D + part * 4);
            if (p.decay_row && !p.s_code) cp_async16(stg + G::sS + tau * D * 4 + part * 16, p.s + tok * D + part * 4);
        }
        if (p.decay_row && p.s_code) {
            for (int c = tt; c < nb * (D / 16); c += 128) {
                const int tau = c / (D / 16), part = c % (D / 16);
                const size_t tok = (tokb + tb + tau) * p.H + h;
                cp_async16(stg + G::sS + tau * D + part * 16, p.s_code + tok * D + part * 16);
            }
        } else if (!p.decay_row && tt < nb) {
            const size_t tok = (tokb + tb + tt) * p.H + h;
            if (p.s_code)   // one code per head and token: its level, stored directly
                reinterpret_cast<float*>(stg + G::sS)[tt] =
                    __ldg(p.s_lut + static_cast<size_t>(h) * p.L + min(static_cast<int>(p.s_code[tok]), p.L - 1));
            else
                cp_async4(stg + G::sS + tt * 4, p.s + tok);
        }
        cp_async_commit();
    };
    // ... and v, into the row-major state buffer, which is free between the state's way in and
    // the last block's way out (global loads in flight would hold up every barrier)
    auto issue_v = [&](int tb) {
        const int nb = min(L, p.t_end - tb);
        for (int c = tt; c < nb * (D / 4); c += 128) {
            const int tau = c / (D / 4), part = c % (D / 4);
            cp_async16(sbuf + tau * D + part * 4, p.v + ((tokb + tb + tau) * p.H + h) * D + part * 4);
        }
        cp_async_commit();
    };
    if (tt >= 0 && p.t_begin < p.t_end) issue_kqs(p.t_begin);

    // state in: S^T into TMEM (FP32 and lo); this thread's lane j, key rows of its half
#pragma unroll 1
    for (int i0 = 64 * hf; i0 < 64 * hf + 64; i0 += 16) {
        float x[16], lo[16];
#pragma unroll
        for (int c = 0; c < 16; ++c) {
            x[c] = sbuf[sb_off<D>(i0 + c, jl >> 2) + (jl & 3)];
            lo[c] = __fsub_rn(x[c], tc::tf32_hi(x[c]));
        }
        tc::tmem_st16(tl + G::kHi + i0, x);
        tc::tmem_st16(tl + G::kLo + i0, lo);
    }
    tc::wait_st();
    tc::fence_before_sync();

    // Rows: thread (i, half hh) takes tokens 8 hh .. 8 hh + 7 of key row i.  Phase A (staged
    // loads, decays, EMA terms, the first half's EMA recursion) of block c + 1 runs while the
    // tensor cores work on block c; phase B (the second half's EMA recursion, cumulative decays,
    // operand tiles) at the start of block c + 1.  The halves exchange through shared memory the
    // first half's decay product and EMA state and the second half's decay product.
    constexpr int LH = L / 2;
    const int i = tid & (D - 1), hh = tid >> 7, tb = LH * hh;
    float4* xch = reinterpret_cast<float4*>(cb + G::oXch);
    struct RowA {
        float kk[LH], dd[LH], qv[LH], bv[LH], xs[LH], xr[LH];
    };
    auto phase_a = [&](int t0b, RowA& r) {
        const int nb = min(L, p.t_end - t0b);
        const float* sbeta = reinterpret_cast<const float*>(stg + G::sB) + (((t0b - p.t_begin) / L) % 3) * L;
        // branch-free over the half's tokens (tokens past nb read staged bytes of earlier
        // blocks, in bounds, and are masked), so the eight exp / expm1 chains interleave
        bool bad = false;
#pragma unroll
        for (int j = 0; j < LH; ++j) {
            const int tau = tb + j;
            const bool live = tau < nb;
            float rate;
            if (!p.decay_row) {
                rate = ss[tau];
            } else if (p.s_code) {
                const int code = min(static_cast<int>(sc[tau * D + i]), p.L - 1);
                rate = p.L <= 4 ? S.lut[i * p.L + code]
                                : __ldg(p.s_lut + (static_cast<size_t>(h) * D + i) * p.L + code);
            } else {
                rate = ss[tau * D + i];
            }
            bad |= live && (!(rate > 0.0f) || !(rate < INFINITY));
            rate = live ? rate : 1.0f;
            const float kq = sk[tau * D + i], qq = sq[tau * D + i];
            const float bq = p.erase ? sbeta[tau] : 0.0f;
            r.kk[j] = live ? kq : 0.0f;
            r.qv[j] = live ? qq : 0.0f;
            r.bv[j] = live ? bq : 0.0f;
            const float d = expf(-rate);
            r.dd[j] = live ? d : 1.0f;
            r.xs[j] = r.xr[j] = 0.0f;
            if (stats) {
                r.xs[j] = -expm1f(-2.0f * rate);
                r.xr[j] = p.erase ? __fmul_rn(__fmul_rn(r.bv[j], __fsub_rn(2.0f, r.bv[j])), __fmul_rn(r.kk[j], r.kk[j])) : 0.0f;
            }
        }
        if (bad) raise_status(p.status, QS_DEV_RATE);
        float prod = 1.0f;
#pragma unroll
        for (int j = 0; j < LH; ++j) prod = __fmul_rn(prod, r.dd[j]);
        if (hh == 0) {
            // the EMA recursion over the first half (from the state after the previous block)
            float ms = stats ? S.ms[i] : 0.0f, mr = stats ? S.mr[i] : 0.0f;
            if (stats) {
#pragma unroll
                for (int j = 0; j < LH; ++j) {
                    if (j >= nb) break;
                    if (t0b + j == 0) {
                        ms = r.xs[j];
                        mr = r.xr[j];
                    } else {
                        ms = __fadd_rn(ms, __fmul_rn(p.alpha, __fsub_rn(r.xs[j], ms)));
                        mr = __fadd_rn(mr, __fmul_rn(p.alpha, __fsub_rn(r.xr[j], mr)));
                    }
                }
            }
            xch[i] = make_float4(prod, ms, mr, 0.0f);
        } else {
            xch[D + i].x = prod;
        }
    };
    auto phase_b = [&](int t0b, const RowA& r) {
        const int nb = min(L, p.t_end - t0b);
        float* dl = dall + (((t0b - p.t_begin) / L) & 1) * D;
        float pr[LH], sf[LH];
        float acc = 1.0f;
#pragma unroll
        for (int j = 0; j < LH; ++j) pr[j] = acc = __fmul_rn(acc, r.dd[j]);
        acc = 1.0f;
#pragma unroll
        for (int j = LH - 1; j >= 0; --j) {
            sf[j] = acc;
            acc = __fmul_rn(acc, r.dd[j]);
        }
        const float4 x0 = xch[i];
        const float dc0 = hh == 0 ? 1.0f : x0.x;            // decay before the half
        const float sf1 = hh == 0 ? xch[D + i].x : 1.0f;   // decay after the half, in the block
        if (hh == 1) {
            // the EMA state after the whole block and the block's decay (with no second-half
            // tokens, the first half's)
            float ms = x0.y, mr = x0.z;
            if (stats) {
#pragma unroll
                for (int j = 0; j < LH; ++j) {
                    if (tb + j >= nb) break;
                    ms = __fadd_rn(ms, __fmul_rn(p.alpha, __fsub_rn(r.xs[j], ms)));
                    mr = __fadd_rn(mr, __fmul_rn(p.alpha, __fsub_rn(r.xr[j], mr)));
                }
                S.ms[i] = ms;
                S.mr[i] = mr;
            }
            const float Dall = __fmul_rn(dc0, pr[LH - 1]);
            if (!(Dall >= 1e-37f)) raise_status(p.status, QS_DEV_CHUNK);
            dl[i] = Dall;
        }
        const int oh = (i >> 2) * G::kLboH + (i & 3) * 4, ow = (i >> 2) * G::kLboW + (i & 3) * 4;
#pragma unroll
        for (int j = 0; j < LH; ++j) {
            const int tau = tb + j;
            const float Dc = __fmul_rn(dc0, pr[j]);
            const float a = p.erase ? __fmul_rn(r.bv[j], r.kk[j]) : 0.0f;
            const float kt = __fmul_rn(a, Dc), qt = __fmul_rn(r.qv[j], Dc);
            float rDc;   // k / Dc only enters A and M
            asm("rcp.approx.ftz.f32 %0, %1;" : "=f"(rDc) : "f"(Dc));
            const float kh = tau < nb ? __fmul_rn(r.kk[j], rDc) : 0.0f;
            // tiles: k / Dc row tau; [a o Dc ; q o Dc] rows tau and L + tau (row r of a
            // K-chunk at byte 16 r)
            const float khh = tc::tf32_hi(kh), kth = tc::tf32_hi(kt), qth = tc::tf32_hi(qt);
            *reinterpret_cast<float*>(kh_hi + oh + 16 * tau) = khh;
            *reinterpret_cast<float*>(kh_lo + oh + 16 * tau) = __fsub_rn(kh, khh);
            *reinterpret_cast<float*>(bw_hi + ow + 16 * tau) = kth;
            *reinterpret_cast<float*>(bw_lo + ow + 16 * tau) = __fsub_rn(kt, kth);
            *reinterpret_cast<float*>(bw_hi + ow + 16 * (L + tau)) = qth;
            *reinterpret_cast<float*>(bw_lo + ow + 16 * (L + tau)) = __fsub_rn(qt, qth);
        }
        // (k o Dc_{L-1} / Dc)^T: row i, tokens of the half, 4 per 16-byte chunk
#pragma unroll
        for (int c4 = 0; c4 < LH / 4; ++c4) {
            float kb[4];
#pragma unroll
            for (int e = 0; e < 4; ++e) kb[e] = __fmul_rn(r.kk[4 * c4 + e], __fmul_rn(sf[4 * c4 + e], sf1));
            float4 hi, lo;
            hi.x = tc::tf32_hi(kb[0]);
            hi.y = tc::tf32_hi(kb[1]);
            hi.z = tc::tf32_hi(kb[2]);
            hi.w = tc::tf32_hi(kb[3]);
            lo.x = __fsub_rn(kb[0], hi.x);
            lo.y = __fsub_rn(kb[1], hi.y);
            lo.z = __fsub_rn(kb[2], hi.z);
            lo.w = __fsub_rn(kb[3], hi.w);
            const int o = ((tb >> 2) + c4) * G::kLboU + (i >> 3) * G::kSboU + (i & 7) * 16;
            *reinterpret_cast<float4*>(bu_hi + o) = hi;
            *reinterpret_cast<float4*>(bu_lo + o) = lo;
        }
    };

    RowA ra;   // phase A of the block about to start
    if (p.t_begin < p.t_end) {
        if (tt >= 0) cp_async_wait_all();
        __syncthreads();                      // the first block's inputs; the state buffer is read
        if (tt >= 0) issue_v(p.t_begin);
        phase_a(p.t_begin, ra);
        __syncthreads();                      // the first block's exchange; its staging is read
        if (tt >= 0 && p.t_begin + L < p.t_end) issue_kqs(p.t_begin + L);
    }

#pragma unroll 1
    for (int t0 = p.t_begin; t0 < p.t_end; t0 += L) {
        const int n = min(L, p.t_end - t0);
        const bool last = t0 + L >= p.t_end;
        const float* sbeta = reinterpret_cast<const float*>(stg + G::sB) + (((t0 - p.t_begin) / L) % 3) * L;
        const float* dall_c = dall + (((t0 - p.t_begin) / L) & 1) * D;
        phase_b(t0, ra);
        // the next block's k, q, rates and beta and this block's v have landed
        if (tt >= 0) cp_async_wait_all();
        tc::fence_async_smem();
        __syncthreads();                                                            // C1

        // On the tensor cores (3xTF32, K = 128 key rows), issued by two threads of different
        // warps (an issuing thread stalls while the product queue is full): thread 0 issues
        // S_b^T [a o Dc ; q o Dc]^T, its hi*hi product and the two corrections in separate
        // accumulators; thread 32 issues (k / Dc) [a o Dc ; q o Dc]^T, whose row s, column t is
        // A_ts (column < L) or M_ts (column >= L)
        if (tid == 0 || tid == 32) {
            tc::fence_after_sync();
            constexpr uint32_t idW = tc::idesc_tf32(128, 2 * L);
            // A and M need rows 0..L-1 of the product only: M = 64 (rows 0..15 land in lanes 0..15)
            constexpr uint32_t idAM = tc::idesc_tf32(64, 2 * L);
            // a K-step advances the start addresses (16-byte units, bits 0-13) by two K-chunks
            constexpr uint64_t kStepW = (2 * G::kLboW) >> 4, kStepH = (2 * G::kLboH) >> 4;
            uint64_t bh = tc::smem_desc(tc::smem_addr(bw_hi), G::kLboW, G::kSboW);
            uint64_t bl = tc::smem_desc(tc::smem_addr(bw_lo), G::kLboW, G::kSboW);
            if (tid == 0) {
#pragma unroll
                for (int ks = 0; ks < D / 8; ++ks) {
                    const uint32_t acc = ks > 0 ? 1u : 0u;
                    tc::mma_tf32_ts(tmem + G::kDW, tmem + G::kHi + 8 * ks, bh, idW, acc);
                    tc::mma_tf32_ts(tmem + G::kDWc, tmem + G::kHi + 8 * ks, bl, idW, acc);
                    tc::mma_tf32_ts(tmem + G::kDWc, tmem + G::kLo + 8 * ks, bh, idW, 1u);
                    bh += kStepW;
                    bl += kStepW;
                }
            } else {
                uint64_t ah = tc::smem_desc(tc::smem_addr(kh_hi), G::kLboH, G::kSboH);
                uint64_t al = tc::smem_desc(tc::smem_addr(kh_lo), G::kLboH, G::kSboH);
#pragma unroll
                for (int ks = 0; ks < D / 8; ++ks) {
                    const uint32_t acc = ks > 0 ? 1u : 0u;
                    tc::mma_tf32_ss(tmem + G::kAM, ah, bh, idAM, acc);
                    tc::mma_tf32_ss(tmem + G::kAMc, ah, bl, idAM, acc);
                    tc::mma_tf32_ss(tmem + G::kAMc, al, bh, idAM, 1u);
                    bh += kStepW;
                    bl += kStepW;
                    ah += kStepH;
                    al += kStepH;
                }
            }
            tc::mma_commit(bar);
        }
        // while the tensor cores work: phase A of the next block
        if (!last) phase_a(t0 + L, ra);
        wait_mma(0);
        if (warp == 0) {
            // A and M to shared memory (lane s < L holds row s of the product): the hi*hi
            // accumulator plus the corrections' (one FP32 rounding)
            float x[L], y[L], xc[L], yc[L];
            tc::tmem_ld2x16(tl + G::kAM, tl + G::kAM + L, x, y);
            tc::tmem_ld2x16(tl + G::kAMc, tl + G::kAMc + L, xc, yc);
            if (lane < L) {
#pragma unroll
                for (int t = 0; t < L; ++t) {
                    amA[t * L + lane] = __fadd_rn(x[t], xc[t]);
                    amM[t * L + lane] = __fadd_rn(y[t], yc[t]);
                }
            }
        }
        __syncthreads();                                                            // C2
        // every thread is done with the next block's staged inputs: the one after it
        if (tt >= 0 && t0 + 2 * L < p.t_end) issue_kqs(t0 + 2 * L);

        if (hf == 1) {
            // u of column j, token by token: u_t = w_t v_t - (S_b^T (a o Dc))_t - sum_{s<t} A_ts u_s
            float wk[L], ck[L];
            tc::tmem_ld2x16(tl + G::kDW, tl + G::kDWc, wk, ck);
            float u[L];
#pragma unroll
            for (int t = 0; t < L; ++t) {
                float pp = __fadd_rn(wk[t], ck[t]);
                // row t of A, four entries per load
#pragma unroll
                for (int s4 = 0; s4 < t; s4 += 4) {
                    const float4 a4 = reinterpret_cast<const float4*>(amA + t * L)[s4 / 4];
                    const float av[4] = {a4.x, a4.y, a4.z, a4.w};
#pragma unroll
                    for (int e = 0; e < 4; ++e)
                        if (s4 + e < t) pp = fmaf(av[e], u[s4 + e], pp);
                }
                const float bt = p.erase ? sbeta[t] : 1.0f;
                const float vj = sbuf[t * D + jl];
                u[t] = t < n ? (p.erase ? __fsub_rn(__fmul_rn(bt, vj), pp) : vj) : 0.0f;
            }
            float uh[L], ul[L];
#pragma unroll
            for (int t = 0; t < L; ++t) {
                uh[t] = tc::tf32_hi(u[t]);
                ul[t] = __fsub_rn(u[t], uh[t]);
            }
            tc::tmem_st16(tl + G::kUHi, uh);
            tc::tmem_st16(tl + G::kULo, ul);
            tc::wait_st();
        }
        tc::fence_before_sync();
        __syncthreads();                                                            // C3
        if (tt >= 0 && !last) issue_v(t0 + L);   // the solve is done with this block's v

        // update = u^T (k o Dc_{L-1} / Dc) on the tensor cores (3xTF32, K = 16 tokens)
        if (tid == 0) {
            tc::fence_after_sync();
            constexpr uint32_t idU = tc::idesc_tf32(128, D);
            constexpr uint64_t kStepU = (2 * G::kLboU) >> 4;
            uint64_t bh = tc::smem_desc(tc::smem_addr(bu_hi), G::kLboU, G::kSboU);
            uint64_t bl = tc::smem_desc(tc::smem_addr(bu_lo), G::kLboU, G::kSboU);
#pragma unroll
            for (int ks = 0; ks < L / 8; ++ks) {
                tc::mma_tf32_ts(tmem + G::kUpd, tmem + G::kUHi + 8 * ks, bh, idU, ks > 0 ? 1u : 0u);
                tc::mma_tf32_ts(tmem + G::kUpd, tmem + G::kUHi + 8 * ks, bl, idU, 1u);
                tc::mma_tf32_ts(tmem + G::kUpd, tmem + G::kULo + 8 * ks, bh, idU, 1u);
                bh += kStepU;
                bl += kStepU;
            }
            tc::mma_commit(bar + 1);
        }
        {
            // readouts of column j: o_t = (S_b^T (q o Dc))_t + sum_{s<=t} M_ts u_s, with u from
            // its hi / lo parts in TMEM; warps 0-3 take tokens 0..7 (fewer products: warp 0 also
            // issues the update), warps 4-7 tokens 8..15 of the same columns (the same TMEM lanes)
            float wq[L], cq[L], u[L], ul[L];
            tc::tmem_ld2x16(tl + G::kDW + L, tl + G::kDWc + L, wq, cq);
            tc::tmem_ld2x16(tl + G::kUHi, tl + G::kULo, u, ul);
#pragma unroll
            for (int t = 0; t < L; ++t) u[t] = __fadd_rn(u[t], ul[t]);
#pragma unroll
            for (int t = 0; t < L; ++t) {
                if ((t >= L / 2) != (hf == 1)) continue;
                float oa = __fadd_rn(wq[t], cq[t]), ob = 0.0f;
                // row t of M, four entries per load
#pragma unroll
                for (int s4 = 0; s4 <= t; s4 += 4) {
                    const float4 m4 = reinterpret_cast<const float4*>(amM + t * L)[s4 / 4];
                    if (s4 <= t) oa = fmaf(m4.x, u[s4], oa);
                    if (s4 + 1 <= t) ob = fmaf(m4.y, u[s4 + 1], ob);
                    if (s4 + 2 <= t) oa = fmaf(m4.z, u[s4 + 2], oa);
                    if (s4 + 3 <= t) ob = fmaf(m4.w, u[s4 + 3], ob);
                }
                if (t < n) p.o[((tokb + t0 + t) * p.H + h) * D + jl] = oa + ob;
            }
        }
        wait_mma(1);
        // S_e = fma(S_b, Dc_{L-1}, update): to TMEM (with its lo) for the next block, or, after
        // the interval's last block, to the row-major buffer
#pragma unroll 1
        for (int c0 = 64 * hf; c0 < 64 * hf + 64; c0 += 16) {
            float x[16], up[16], lo[16];
            tc::tmem_ld2x16(tl + G::kHi + c0, tl + G::kUpd + c0, x, up);
#pragma unroll
            for (int c = 0; c < 16; ++c) {
                x[c] = fmaf(x[c], dall_c[c0 + c], up[c]);
                if (last) sbuf[sb_off<D>(c0 + c, jl >> 2) + (jl & 3)] = x[c];
                else lo[c] = __fsub_rn(x[c], tc::tf32_hi(x[c]));
            }
            if (!last) {
                tc::tmem_st16(tl + G::kHi + c0, x);
                tc::tmem_st16(tl + G::kLo + c0, lo);
            }
        }
        if (!last) tc::wait_st();
        tc::fence_before_sync();
    }
    if (p.t_begin >= p.t_end) {
        // no tokens: the state goes back unchanged
#pragma unroll 1
        for (int i0 = 64 * hf; i0 < 64 * hf + 64; i0 += 16) {
            float x[16];
            tc::tmem_ld16(tl + G::kHi + i0, x);
#pragma unroll
            for (int c = 0; c < 16; ++c) sbuf[sb_off<D>(i0 + c, jl >> 2) + (jl & 3)] = x[c];
        }
    }
}

}  // namespace qs
