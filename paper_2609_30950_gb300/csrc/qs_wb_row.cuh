// qs_wb_row.cuh -- persistent write-back kernel for the row allocation unit (sm_103a).
//
// The hot path of qstate_step / qstate_scan for per-row widths (KDA, Mamba-2): one write-back
// interval of every head, packed state in, packed state out.
//
// Each CTA (NW = 8 warps, two CTAs per SM so that one's barriers and latencies overlap the
// other's work) walks a contiguous block of heads.  While it works on head g, cp.async copies
// head g + 1's metadata into the other half of a double buffer (widths in/out, FP16 scales,
// fitted-factor indices, EMA statistics, the first token's k, q, v, rates and their level
// table; issued by the one warp without a prep role) and, once head g's tokens are done, head
// g + 1's packed rows into the single payload buffer (their byte window comes from offsets
// fetched one head earlier).
//
// Two thread layouts share the head's FP32 state:
//  * update layout: warp w owns key rows [w RPW, (w+1) RPW), lane l the value columns
//    [l CPL, (l+1) CPL), so the reductions of Eq. (1) over key rows stay in registers.  The
//    packed rows are decoded straight into it (each lane reads its CPL codes at bit
//    l CPL w of the row, for any width w).
//  * row layout: TPR = dv/32 lanes per row, each owning 32 consecutive value columns, i.e. a
//    word-aligned run of 32 codes (4w bytes).  Warps take rows in order of output width (a
//    sort per head), so the code arithmetic of a warp is specialised for one width.
//    Used for the write-back (range, factor search, codes, packing); the state reaches it
//    through a shared-memory buffer (16-byte groups XOR-swizzled per row).
// Per head there are six CTA barriers:
//   B1  the head's inputs have landed            -> prep, one role per warp group: row offsets
//       (prefix sums of widths) and layout checks; per-row decay, EMA update, dequantisation
//       constants with the first token's decay folded in, erase vector, k.q; rows sorted by
//       output width; and, on the last warp, the next head's metadata copies
//   B2  -> unpack into registers (update layout),
//       partials p = a^T S', r = q^T S'
//   B3  -> u = beta v - p, o = r + u (k.q); meanwhile the next token's inputs are prepared
//       in a second buffer (from registers loaded one more token ahead)
//   B4  -> S = S' + k u^T.  Further tokens of the interval repeat from the partials, so each
//       token costs two barriers.  Then the next head's packed rows are copied in and the
//       state goes to the shared buffer
//   B5  -> write-back (row layout), batches of rows claimed dynamically: row range R, the 16
//       candidate steps and their squared errors (refit), codes, and each lane's packed
//       words stored to the output region
//   B6  -> coalesced stores of scales, factor indices, ranges and EMAs.
// The next head's B1 orders the reuse of stage and staging buffers.
#pragma once

#include <algorithm>

#include "qs_common.cuh"
#include "qs_chunk.cuh"   // the chunked form of the interval

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
    float lut[DK * 4];                           // the head's decay levels (when 2^g <= 4)
    float ga[DK], gw[DV];                        // general erasure: the first token's a and w
    float beta, rate_h, pad0, pad1;
    int in_off, in_end, out_off, ok;              // payload window of this head
    int nxt_in_off, nxt_in_end, nxt_out_off, pad2;   // offsets of the following head
};

template <int DK, int DV, int NW>
struct WbGeom {
    static constexpr int RPW = DK / NW;       // update layout: rows per warp
    static constexpr int CPL = DV / 32;       // update layout: columns per lane
    static constexpr int TPR = DV / 32;       // row layout: lanes per row
    static constexpr int RPB = 32 / TPR;      // row layout: rows per warp
    static constexpr int KPT = kNFit / TPR;   // candidate steps each lane of a row prepares
};

template <int DK, int DV, int NW>
struct alignas(16) WbSmem {
    WbStage<DK, DV> st[2];
    float sbuf[DK * DV];                  // FP32 state of the head (swizzled rows)
    union {
        float red[2][NW][DV];             // p and r partials per warp (token phase)
        float2 cand[NW][32 / (DV / 32)][kNFit + 1];   // per warp and row: (1/Delta_k, -Delta_k)
                                                      // (rows padded against bank conflicts)
        int hist[17 * kNFit + 16];        // prep: counting sort of the rows (width, factor)
    } rc;
    float4 deqAS[DK];                     // (-A, -A, S, S) and (B, B): x = (2^23 + u - A) S + B,
    float2 deqB[DK];                      // as pairs, the operands of packed FP32 arithmetic
    float4 wc[17];                        // per width: (n, 1/n, 2^23*1.5 - n, 2^23*1.5 + n)
    // token inputs, double-buffered by token parity (C > 1; k triple-buffered by token index
    // mod 3).  Buffer 0 of the head's first token is the stage (k, q, v, w) with a and d here;
    // later tokens alternate between buffer 1 (tk, tq, tv, tw, a1, d1) and buffer 0 (the
    // stage's arrays, a, d); k takes the stage, tk and tk2 in turn.
    float tk[DK], tk2[DK], tq[DK], tv[DV];
    float tw[DV];                         // general erasure: w
    float a[DK], d[DK];                   // erase vector a (beta k), decay (buffer 0)
    float a1[DK], d1[DK];                 // (buffer 1)
    float tbeta[2];
    float u[DV];
    float rowR[DK];
    float fitf[kNFit];
    float wsum[2][NW];                    // k.q partials per warp of rows, by buffer
    alignas(16) int off_in[DK + 4];
    alignas(16) int off_out[DK + 4];
    uint8_t ord_out[DK];                  // rows in order of output width
    uint16_t out_scale[DK];
    uint8_t out_fidx[DK];
    int flag;
    int bat_next;                         // next row batch of the write-back to claim
};

// Float offset of 16-byte group G of row i in the state buffer.  The XOR keeps each group in
// its block of 8 and spreads, over the 32 banks, the groups that one 8-lane phase touches in
// the update layout (one row) and, for two rows of different parity, in the row layout.
template <int DV>
__device__ __forceinline__ int sb_off(int i, int G) {
    int s;
    if constexpr (DV == 128) s = ((G >> 3) & 3) | ((i & 1) << 2);
    else s = ((G >> 3) & 1) | ((i & 3) << 1);
    return i * DV + 4 * (G ^ s);
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

// Decoding in the update layout: a lane's CPL codes of a row of width w (up to 16) at bit
// lane CPL w, without a branch on the width: three words are read and the lane's bits taken
// from their 64-bit window, so the decoding of consecutive rows of different
// widths can overlap.  `row` is followed by >= 12 readable bytes.
template <int CPL>
__device__ __forceinline__ void extract_codes_flat(const uint8_t* row, int lane, int w,
                                                   uint32_t (&u)[CPL]) {
    const uint32_t* words = reinterpret_cast<const uint32_t*>(row);
    const int P = lane * CPL * w;
    const int idx = P >> 5, sh = P & 31;
    const uint32_t mask = (1u << w) - 1u;
    const uint32_t lo = __funnelshift_r(words[idx], words[idx + 1], sh);
    const uint32_t hi = __funnelshift_r(words[idx + 1], words[idx + 2], sh);
    const uint64_t chunk = (static_cast<uint64_t>(hi) << 32) | lo;
#pragma unroll
    for (int c = 0; c < CPL; ++c) u[c] = static_cast<uint32_t>(chunk >> (c * w)) & mask;
}

// ---- row layout: 32 consecutive codes of one row per lane ---------------------------------------
// The lane's codes occupy the 4W bytes at byte 4 W q of the row (q = its part), a whole number of
// words: code c of the run sits at bits [c W, c W + W) of those words.

// Packing.  With t_c = fl(x_c / Delta) + kMagic (round to nearest even; its bit pattern is
// kMagicBits + q_c), the stored code u_c = clamp(q_c + n, 0, 2n) is one add-min-relu on the bits;
// codes are shifted into the lane's words (codes that straddle two words add their high bits to
// the next word).
template <int W, int C>
__device__ __forceinline__ void run_put(uint32_t (&wd)[W], uint32_t u) {
    constexpr int bp = C * W, k = bp >> 5, sh = bp & 31;
    wd[k] += u << sh;
    if constexpr (sh + W > 32) wd[k + 1] += u >> (32 - sh);
}

template <int W, int C>
struct RunEncode {
    __device__ __forceinline__ static void go(uint32_t (&wd)[W], const float2 (&xv)[16], float2 i2, int off, int top) {
        const float2 t = __fadd2_rn(__fmul2_rn(xv[C / 2], i2), make_float2(kMagic, kMagic));
        run_put<W, C>(wd, static_cast<uint32_t>(__viaddmin_s32_relu(__float_as_int(t.x), off, top)));
        run_put<W, C + 1>(wd, static_cast<uint32_t>(__viaddmin_s32_relu(__float_as_int(t.y), off, top)));
        RunEncode<W, C + 2>::go(wd, xv, i2, off, top);
    }
};
template <int W>
struct RunEncode<W, 32> {
    __device__ __forceinline__ static void go(uint32_t (&)[W], const float2 (&)[16], float2, int, int) {}
};

// MAXA: alignment of the row starts (16 bytes for dv = 128, 8 for dv = 64).
template <int NWD, int MAXA>
__device__ __forceinline__ void store_words(uint8_t* dst, const uint32_t (&wd)[NWD]) {
    if constexpr (NWD % 4 == 0 && MAXA >= 16) {
#pragma unroll
        for (int k = 0; k < NWD; k += 4)
            *reinterpret_cast<uint4*>(dst + 4 * k) = make_uint4(wd[k], wd[k + 1], wd[k + 2], wd[k + 3]);
    } else if constexpr (NWD % 2 == 0) {
#pragma unroll
        for (int k = 0; k < NWD; k += 2) *reinterpret_cast<uint2*>(dst + 4 * k) = make_uint2(wd[k], wd[k + 1]);
    } else {
#pragma unroll
        for (int k = 0; k < NWD; ++k) reinterpret_cast<uint32_t*>(dst)[k] = wd[k];
    }
}

// Quantise + pack the lane's 32 values (row of width W) to dst (4W bytes at byte 4 W q of a row
// aligned to MAXA bytes): q = clamp(rint(x / Delta), -n, n), offset binary.
template <int W, int MAXA>
__device__ __forceinline__ void pack_run(const float2 (&xv)[16], float inv, uint8_t* dst) {
    if constexpr (W == 1) {
        // sign bit, code 1 for x < 0 (negative zero counts as positive)
        uint32_t wd[1] = {0u};
#pragma unroll
        for (int c = 0; c < 16; ++c) {
            wd[0] |= (xv[c].x < 0.0f ? 1u : 0u) << (2 * c);
            wd[0] |= (xv[c].y < 0.0f ? 2u : 0u) << (2 * c);
        }
        store_words<1, MAXA>(dst, wd);
    } else if constexpr (W >= 2) {
        constexpr int n = (1 << (W - 1)) - 1;
        uint32_t wd[W];
#pragma unroll
        for (int k = 0; k < W; ++k) wd[k] = 0u;
        RunEncode<W, 0>::go(wd, xv, make_float2(inv, inv), n - static_cast<int>(kMagicBits), 2 * n);
        store_words<W, MAXA>(dst, wd);
    }
}

template <int MAXA>
__device__ __forceinline__ void pack_row(int w, const float2 (&xv)[16], float inv, uint8_t* dst) {
    switch (w) {
#define QS_W(N) case N: pack_run<N, MAXA>(xv, inv, dst); break;
        QS_W(1) QS_W(2) QS_W(3) QS_W(4) QS_W(5) QS_W(6) QS_W(7) QS_W(8)
        QS_W(9) QS_W(10) QS_W(11) QS_W(12) QS_W(13) QS_W(14) QS_W(15) QS_W(16)
#undef QS_W
        default: break;
    }
}

// Issue the asynchronous copies of head g's metadata into stage S, by threads t = 0..nt-1 of
// the calling group (the whole CTA for a CTA's first head; one warp, which has no other work in
// the prep phase, for the heads after it).  The head's payload window (in_off, in_end) and output
// offset come from the previous stage (or, for the first head, from direct loads) and are checked
// here; gnext >= 0 names the head whose offsets to fetch.  One commit group per call.
template <int DK, int DV>
__device__ __forceinline__ void wb_issue_meta(WbStage<DK, DV>& S, int g, int gnext, int in_off, int in_end,
                                           int out_off, const WbParams& wp, int t, int nt) {
    const StepParams& p = wp.s;
    const bool stats = p.ema_s != nullptr;
    const int T = p.T;
    const int b = g / p.H, h = g - (g / p.H) * p.H;
    const size_t tok = (static_cast<size_t>(b) * T + p.t_begin) * p.H + h;
    const size_t rb = static_cast<size_t>(g) * DK;
    // one array at a time, in 16-byte chunks
    auto seg = [&](void* dst, const void* src, int nchunks) {
        for (int c = t; c < nchunks; c += nt)
            cp_async16(static_cast<uint8_t*>(dst) + 16 * c, static_cast<const uint8_t*>(src) + 16 * c);
    };
    constexpr int C8 = DK / 16, C16 = DK * 2 / 16, C32 = DK * 4 / 16, CV = DV * 4 / 16;
    seg(S.w_in, p.in_widths + rb, C8);
    seg(S.w_out, p.out_widths + rb, C8);
    seg(S.fidx, p.in_fidx + rb, C8);
    seg(S.sc_in, p.in_scales + rb, C16);
    seg(S.k, p.k + tok * DK, C32);
    seg(S.q, p.q + tok * DK, C32);
    seg(S.v, p.v + tok * DV, CV);
    if (stats) {
        seg(S.ms, p.ema_s + rb, C32);
        seg(S.mr, p.ema_r + rb, C32);
    }
    if (p.decay_row && !p.s_code) seg(S.s, p.s + tok * DK, C32);
    if (p.decay_row && p.s_code) seg(S.scode, p.s_code + tok * DK, C8);
    // general erasure: the first token's a (DK floats) and w (DV floats)
    if (p.general) {
        seg(S.ga, p.a_in + tok * DK, DK / 4);
        seg(S.gw, p.w_in + tok * DV, DV / 4);
    }
    // the head's decay levels (DK x L floats) when L <= 4
    if (p.decay_row && p.s_code && p.L <= 4) seg(S.lut, p.s_lut + static_cast<size_t>(h) * DK * p.L, DK * p.L / 4);
    // scalars and the offsets of the next head
    if (t == nt - 1) {
        if (p.erase) cp_async4(&S.beta, p.beta + tok);
        if (!p.decay_row && !p.s_code) cp_async4(&S.rate_h, p.s + tok);
    }
    const bool next_last = gnext >= 0 && gnext - (gnext / p.H) * p.H == p.H - 1;
    if (t == nt - 2 && gnext >= 0) {
        cp_async4(&S.nxt_in_off, p.in_head_off + gnext);
        cp_async4(&S.nxt_out_off, p.out_head_off + gnext);
        if (!next_last) cp_async4(&S.nxt_in_end, p.in_head_off + gnext + 1);
    }
    // payload window (copied by wb_issue_payload)
    const int align = DV == 128 ? 16 : 8;
    const int nbytes = in_end - in_off;
    const bool ok = in_off >= 0 && nbytes >= 0 && nbytes <= p.stage_bytes && in_off % align == 0 &&
                    nbytes % align == 0 && static_cast<long long>(in_end) <= p.region_bytes;
    if (t == 0) {
        S.in_off = in_off;
        S.in_end = in_end;
        S.out_off = out_off;
        S.ok = ok ? 1 : 0;
        // the next head's window ends at the head after it (copied above), or at the end of the
        // region for the last head of a batch element
        if (next_last) S.nxt_in_end = static_cast<int>(p.region_bytes);
    }
    cp_async_commit();
}

// Copy head g's packed rows (the window recorded in S by wb_issue_meta; S.ok must be visible
// to every thread) into pay.  One commit group per call.
template <int DK, int DV>
__device__ __forceinline__ void wb_issue_payload(const WbStage<DK, DV>& S, uint8_t* pay, int g, const WbParams& wp) {
    const StepParams& p = wp.s;
    const int tid = threadIdx.x;
    if (S.ok) {
        const int b = g / p.H;
        const int nbytes = S.in_end - S.in_off;
        const uint8_t* src = p.in_payload + static_cast<size_t>(b) * p.region_bytes + S.in_off;
        if (DV == 128) {
            for (int i = tid; i < nbytes / 16; i += blockDim.x) cp_async16(pay + 16 * i, src + 16 * i);
        } else {
            for (int i = tid; i < nbytes / 8; i += blockDim.x) cp_async8(pay + 8 * i, src + 8 * i);
        }
    }
    cp_async_commit();
}

// ---- the kernel ---------------------------------------------------------------------------------
// CHUNK: the interval runs in chunked form on the tensor cores (qs_chunk.cuh; dk = dv = 128),
// one CTA per SM (all of TMEM, about 190 KB of shared memory); otherwise token by token.
template <int DK, int DV, int NW, bool CHUNK = false>
__global__ void __launch_bounds__(NW * 32, CHUNK ? 1 : 2) wb_row_kernel(const WbParams wp) {
    using Geo = WbGeom<DK, DV, NW>;
    constexpr int RPW = Geo::RPW, CPL = Geo::CPL, CP2 = CPL / 2;
    constexpr int TPR = Geo::TPR, RPB = Geo::RPB, KPT = Geo::KPT, NB = DK / RPB;
    static_assert(CPL == 2 || CPL == 4, "value columns");
    static_assert(RPW >= 2 && RPW <= 16 && NW == 8, "warps");
    using Sm = WbSmem<DK, DV, NW>;
    using Stage = WbStage<DK, DV>;
    const StepParams& p = wp.s;
    extern __shared__ __align__(16) uint8_t smem_raw[];
    Sm& sm = *reinterpret_cast<Sm*>(smem_raw);
    uint8_t* pay = smem_raw + sizeof(Sm);
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const bool stats = p.ema_s != nullptr;
    const int T = p.T;

    if (tid < kNFit) sm.fitf[tid] = fit_factor(tid);
    if (tid >= 32 && tid < 32 + 17) {
        const int w = tid - 32;
        const float n = w >= 2 ? static_cast<float>((1 << (w - 1)) - 1) : 0.0f;
        sm.wc[w] = make_float4(n, w >= 2 ? __frcp_rn(n) : 0.0f, kMagic - n, kMagic + n);
    }

    // a contiguous block of heads per CTA
    const int g_begin = static_cast<int>(static_cast<long long>(blockIdx.x) * wp.nheads / gridDim.x);
    const int g_end = static_cast<int>(static_cast<long long>(blockIdx.x + 1) * wp.nheads / gridDim.x);
    if (g_begin >= g_end) return;
    uint8_t* cb = pay + ((p.stage_bytes + 32 + 15) & ~15);   // chunked form's region
    uint32_t tmem = 0, mphase = 0;
    if constexpr (CHUNK) tmem = chunk_setup(cb);
    {
        const int h0 = g_begin % p.H;
        const int io = static_cast<int>(p.in_head_off[g_begin]);
        const int ie = h0 < p.H - 1 ? static_cast<int>(p.in_head_off[g_begin + 1]) : static_cast<int>(p.region_bytes);
        const int oo = static_cast<int>(p.out_head_off[g_begin]);
        wb_issue_meta<DK, DV>(sm.st[0], g_begin, g_begin + 1 < g_end ? g_begin + 1 : -1, io, ie, oo, wp,
                              tid, NW * 32);
        __syncthreads();
        wb_issue_payload<DK, DV>(sm.st[0], pay, g_begin, wp);
    }

    for (int g = g_begin, j = 0; g < g_end; ++g, ++j) {
        const int sidx = j & 1;
        Stage& S = sm.st[sidx];
        const int b = g / p.H, h = g - (g / p.H) * p.H;
        cp_async_wait_all();
        if (tid == 0) sm.flag = S.ok ? 0 : 1;
        __syncthreads();                                                               // B1
        const bool has_next = g + 1 < g_end;
        // the next head's metadata, by the warp that has no prep role
        if (has_next && warp == NW - 1)
            wb_issue_meta<DK, DV>(sm.st[sidx ^ 1], g + 1, g + 2 < g_end ? g + 2 : -1, S.nxt_in_off,
                                  S.nxt_in_end, S.nxt_out_off, wp, lane, 32);

        // ---- prep ---------------------------------------------------------------------------
        const size_t tok0 = (static_cast<size_t>(b) * T + p.t_begin) * p.H + h;
        const float beta0 = p.erase ? S.beta : 1.0f;
        float rate_h = 0.0f;
        if (!p.decay_row)
            rate_h = p.s_code ? __ldg(p.s_lut + static_cast<size_t>(h) * p.L +
                                      min(static_cast<int>(p.s_code[tok0]), p.L - 1))
                              : S.rate_h;
        if (warp < 2) {
            // row byte offsets: exclusive prefix sums of w dv / 8 (warp 0 input, warp 1 output)
            const uint8_t* wa = warp == 0 ? S.w_in : S.w_out;
            int* off = warp == 0 ? sm.off_in : sm.off_out;
            constexpr int PER = DK / 32;
            int loc[PER];
            int sum = 0;
            bool bad = false;
#pragma unroll
            for (int jj = 0; jj < PER; ++jj) {
                const int w = wa[lane * PER + jj];
                bad |= (w > 16) && (warp == 0 || p.mode != 1);   // statistics only: no output rows
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
                else if (p.mode != 1)
                    bad |= (total > p.stage_bytes || S.out_off % align != 0 || S.out_off < 0 ||
                            static_cast<long long>(S.out_off) + total > p.region_bytes);
                if (bad) atomicExch(&sm.flag, 1);
            }
        } else if (tid >= 64 && tid < 64 + DK) {
            const int i = tid - 64;
            const float kk = S.k[i];
            float rate = rate_h;
            if (p.decay_row) {
                if (p.s_code) {
                    const int code = min(static_cast<int>(S.scode[i]), p.L - 1);
                    rate = p.L <= 4 ? S.lut[i * p.L + code]
                                    : __ldg(p.s_lut + (static_cast<size_t>(h) * DK + i) * p.L + code);
                } else {
                    rate = S.s[i];
                }
            }
            if (!(rate > 0.0f) || !(rate < INFINITY)) raise_status(p.status, QS_DEV_RATE);
            const float d = CHUNK ? 1.0f : expf(-rate);   // the chunked form decays every token itself
            const float ai = p.general ? S.ga[i] : __fmul_rn(beta0, kk);
            if (stats && !CHUNK) {
                const float xs = -expm1f(-2.0f * rate);
                float xr = p.erase ? __fmul_rn(__fmul_rn(beta0, __fsub_rn(2.0f, beta0)), __fmul_rn(kk, kk)) : 0.0f;
                if (p.general) xr = general_erasure<DK>(ai, kk, S.k);
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
            const float Sd = (w >= 2 ? D : (w == 1 ? -2.0f * D : 0.0f)) * d, Bd = (w == 1 ? D : 0.0f) * d;
            sm.deqAS[i] = make_float4(-A, -A, Sd, Sd);
            sm.deqB[i] = make_float2(Bd, Bd);
            sm.a[i] = ai;
            // k . q: one partial per warp of rows
            const float kq = warp_sum(kk * S.q[i]);
            if (lane == 0) sm.wsum[0][(tid - 64) >> 5] = kq;
        } else if (warp == 6) {
            // Rows in order of output width, and within a width in order of the factor fitted
            // at the previous write-back (a close predictor of this one's), any order among
            // equals.  Widths 2..16 come first in ascending order (the narrowest rows have the
            // longest range-factor search), then widths 1 and 0; within a width the smaller
            // factors first (the search runs from the largest factor down, so they search
            // longest).  The write-back claims batches of rows in this order: longest first,
            // and the rows of a batch stop their searches at similar candidates.  A counting
            // sort: histogram of the 17 x 16 keys, exclusive scan, ranks from the atomics.
            constexpr int PER = DK / 32, NK = 17 * kNFit, KPL = (NK + 31) / 32;
            int* hist = sm.rc.hist;
            for (int k = lane; k < NK; k += 32) hist[k] = 0;
            __syncwarp();
            int key[PER], rank[PER];
#pragma unroll
            for (int jj = 0; jj < PER; ++jj) {
                const int i = lane * PER + jj;
                key[jj] = ((min(static_cast<int>(S.w_out[i]), 16) + 15) % 17) * kNFit + (S.fidx[i] & (kNFit - 1));
                rank[jj] = atomicAdd(&hist[key[jj]], 1);
            }
            __syncwarp();
            int cnt[KPL], sum = 0;
#pragma unroll
            for (int m = 0; m < KPL; ++m) {
                const int k = lane * KPL + m;
                cnt[m] = sum;
                sum += k < NK ? hist[k] : 0;
            }
            int incl = sum;
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                const int n = __shfl_up_sync(kFull, incl, o);
                if (lane >= o) incl += n;
            }
            __syncwarp();
#pragma unroll
            for (int m = 0; m < KPL; ++m) {
                const int k = lane * KPL + m;
                if (k < NK) hist[k] = incl - sum + cnt[m];
            }
            __syncwarp();
#pragma unroll
            for (int jj = 0; jj < PER; ++jj)
                sm.ord_out[hist[key[jj]] + rank[jj]] = static_cast<uint8_t>(lane * PER + jj);
            if (lane == 0) sm.bat_next = NW;
        }
        __syncthreads();                                                               // B2
        if (sm.flag != 0) {
            if (tid == 0) raise_status(p.status, QS_DEV_LAYOUT);
            if (has_next) wb_issue_payload<DK, DV>(sm.st[sidx ^ 1], pay, g + 1, wp);
            continue;
        }

        // ---- unpack + dequantise into the update layout (first token's decay folded in) -------
        // At dv = 128 lane l holds columns 4l..4l+3 of the warp's RPW rows.  At dv = 64 the two
        // half-warps take alternate rows (RS = 2) and lane l columns 4 (l % 16)..+3, so a lane
        // still decodes four codes per row it visits; the partials are combined across the
        // halves with one shuffle per value.
        constexpr int RS = DV == 128 ? 1 : 2, NSL = RPW / RS;
        const int half = lane / (32 / RS), cl = lane % (32 / RS);
        float2 x[NSL][2];
        if constexpr (RS == 2) {
#pragma unroll
            for (int jr = 0; jr < NSL; ++jr) {
                const int i = warp * RPW + jr * RS + half;
                uint32_t u[4];
                extract_codes_flat<4>(pay + sm.off_in[i], cl, static_cast<int>(S.w_in[i]), u);
                const float4 as = sm.deqAS[i];
                const float2 A2 = make_float2(as.x, as.y), S2 = make_float2(as.z, as.w), B2 = sm.deqB[i];
#pragma unroll
                for (int c = 0; c < 2; ++c) {
                    const float2 t2 = make_float2(__uint_as_float(kTwo23Bits | u[2 * c]),
                                                  __uint_as_float(kTwo23Bits | u[2 * c + 1]));
                    x[jr][c] = __ffma2_rn(__fadd2_rn(t2, A2), S2, B2);
                }
            }
        } else {
#pragma unroll
        for (int r4 = 0; r4 < RPW; r4 += 4) {
            const int i0 = warp * RPW + r4;
            const int4 o4 = *reinterpret_cast<const int4*>(&sm.off_in[i0]);
            const uint32_t w4 = *reinterpret_cast<const uint32_t*>(&S.w_in[i0]);
            const int offs[4] = {o4.x, o4.y, o4.z, o4.w};
#pragma unroll
            for (int rr = 0; rr < 4; ++rr) {
                const int r = r4 + rr;
                uint32_t u[CPL];
                extract_codes_flat<CPL>(pay + offs[rr], lane, static_cast<int>((w4 >> (8 * rr)) & 0xFFu), u);
                const float4 as = sm.deqAS[i0 + rr];
                const float2 A2 = make_float2(as.x, as.y), S2 = make_float2(as.z, as.w), B2 = sm.deqB[i0 + rr];
#pragma unroll
                for (int c = 0; c < CP2; ++c) {
                    const float2 t2 = make_float2(__uint_as_float(kTwo23Bits | u[2 * c]),
                                                  __uint_as_float(kTwo23Bits | u[2 * c + 1]));
                    x[r][c] = __ffma2_rn(__fadd2_rn(t2, A2), S2, B2);
                }
            }
        }
        }

        // ---- tokens of the interval (Eq. 1) ----------------------------------------------------
        // Per token: (A) every warp applies the decay (tokens after the first; the first one's
        // is folded into the dequantisation) and forms the partials p = S'^T a, r = S'^T q; B3;
        // (B) the first DV threads take the column sums, u = w o v - p and o = r + u (k.q),
        // while the last DK threads prepare the next token's inputs (decay, a, statistics, k.q)
        // in the other buffer from raw values loaded into registers one token earlier, and load
        // the raw values of the token after next; B4; (C) S = S' + k u^T (and, under general
        // erasure, the next token's erasure statistic, which needs all of its k).
        constexpr int P0 = NW * 32 - DK;   // first thread of the input-preparing role
        static_assert(P0 >= DV, "the two roles of the middle phase overlap");
        const int pi = tid - P0;
        const bool prep_k = pi >= 0, prep_v = pi >= 0 && pi < DV;
        // A preparing thread holds the raw inputs of one token in registers (its row's k, q,
        // rate or rate code, a; beta; its column's v, w): right after preparing token t + 1 it
        // loads token t + 2's, so the loads have a whole token to arrive.  The per-token stride
        // of every input is H rows.
        float rk = 0.0f, rq = 0.0f, rs = 0.0f, rbeta = 1.0f, rv = 0.0f, ra = 0.0f, rw = 0.0f;
        int rc = 0;
        auto load_raw = [&](size_t tn) {
            rk = __ldg(p.k + tn * DK + pi);
            rq = __ldg(p.q + tn * DK + pi);
            const size_t si = p.decay_row ? tn * DK + pi : tn;
            if (p.s_code) rc = p.s_code[si];
            else rs = __ldg(p.s + si);
            if (p.erase) rbeta = __ldg(p.beta + tn);
            if (p.general) ra = __ldg(p.a_in + tn * DK + pi);
            if (prep_v) {
                rv = __ldg(p.v + tn * DV + pi);
                if (p.general) rw = __ldg(p.w_in + tn * DV + pi);
            }
        };
        if (!CHUNK && prep_k && p.t_begin + 1 < p.t_end) load_raw(tok0 + p.H);
        for (int t = p.t_begin, j = 0; !CHUNK && t < p.t_end; ++t, ++j) {
            const size_t tok = (static_cast<size_t>(b) * T + t) * p.H + h;
            const int cb = j & 1, k3 = j % 3;
            const float* kv = k3 == 0 ? S.k : k3 == 1 ? sm.tk : sm.tk2;
            const float* qv = cb ? sm.tq : S.q;
            const float* av = cb ? sm.a1 : sm.a;
            if (j > 0 && RS == 2) {
                const float* dd = cb ? sm.d1 : sm.d;
#pragma unroll
                for (int jr = 0; jr < NSL; ++jr) {
                    const float d = dd[warp * RPW + jr * RS + half];
                    x[jr][0] = __fmul2_rn(x[jr][0], make_float2(d, d));
                    x[jr][1] = __fmul2_rn(x[jr][1], make_float2(d, d));
                }
            } else if (j > 0) {
                const float* dd = cb ? sm.d1 : sm.d;
#pragma unroll
                for (int r4 = 0; r4 < RPW; r4 += 4) {
                    const float4 d4 = *reinterpret_cast<const float4*>(&dd[warp * RPW + r4]);
                    const float ds[4] = {d4.x, d4.y, d4.z, d4.w};
#pragma unroll
                    for (int j4 = 0; j4 < 4; ++j4) {
                        const float2 d2 = make_float2(ds[j4], ds[j4]);
#pragma unroll
                        for (int c = 0; c < CP2; ++c) x[r4 + j4][c] = __fmul2_rn(x[r4 + j4][c], d2);
                    }
                }
            }
            float2 pp[2], rr[2];
#pragma unroll
            for (int c = 0; c < 2; ++c) pp[c] = rr[c] = make_float2(0.0f, 0.0f);
            if constexpr (RS == 2) {
#pragma unroll
                for (int jr = 0; jr < NSL; ++jr) {
                    const int i = warp * RPW + jr * RS + half;
                    const float a = av[i], qq = qv[i];
#pragma unroll
                    for (int c = 0; c < 2; ++c) {
                        pp[c] = __ffma2_rn(x[jr][c], make_float2(a, a), pp[c]);
                        rr[c] = __ffma2_rn(x[jr][c], make_float2(qq, qq), rr[c]);
                    }
                }
#pragma unroll
                for (int c = 0; c < 2; ++c) {   // the other half-warp's rows
                    pp[c].x += __shfl_xor_sync(kFull, pp[c].x, 16);
                    pp[c].y += __shfl_xor_sync(kFull, pp[c].y, 16);
                    rr[c].x += __shfl_xor_sync(kFull, rr[c].x, 16);
                    rr[c].y += __shfl_xor_sync(kFull, rr[c].y, 16);
                }
                if (half == 0) {
#pragma unroll
                    for (int c = 0; c < 2; ++c) {
                        reinterpret_cast<float2*>(&sm.rc.red[0][warp][cl * 4])[c] = pp[c];
                        reinterpret_cast<float2*>(&sm.rc.red[1][warp][cl * 4])[c] = rr[c];
                    }
                }
            } else {
#pragma unroll
            for (int r4 = 0; r4 < RPW; r4 += 4) {
                const float4 a4 = *reinterpret_cast<const float4*>(&av[warp * RPW + r4]);
                const float4 q4 = *reinterpret_cast<const float4*>(&qv[warp * RPW + r4]);
                const float as[4] = {a4.x, a4.y, a4.z, a4.w}, qs[4] = {q4.x, q4.y, q4.z, q4.w};
#pragma unroll
                for (int j4 = 0; j4 < 4; ++j4) {
                    const float2 a2 = make_float2(as[j4], as[j4]), q2 = make_float2(qs[j4], qs[j4]);
#pragma unroll
                    for (int c = 0; c < CP2; ++c) {
                        pp[c] = __ffma2_rn(x[r4 + j4][c], a2, pp[c]);
                        rr[c] = __ffma2_rn(x[r4 + j4][c], q2, rr[c]);
                    }
                }
            }
#pragma unroll
            for (int c = 0; c < CP2; ++c) {
                reinterpret_cast<float2*>(&sm.rc.red[0][warp][lane * CPL])[c] = pp[c];
                reinterpret_cast<float2*>(&sm.rc.red[1][warp][lane * CPL])[c] = rr[c];
            }
            }
            __syncthreads();                                                           // B3
            if (tid < DV) {
                const int jv = tid;
                float P = 0.0f, Rr = 0.0f;
#pragma unroll
                for (int w = 0; w < NW; ++w) {
                    P += sm.rc.red[0][w][jv];
                    Rr += sm.rc.red[1][w][jv];
                }
                float kq = 0.0f;
#pragma unroll
                for (int w = 0; w < DK / 32; ++w) kq += sm.wsum[cb][w];
                const float vj = (cb ? sm.tv : S.v)[jv];
                const float beta = j == 0 ? beta0 : sm.tbeta[cb];
                // u = w o v - p (w = beta 1 for the delta rule; a = 0, w = 1 without erasure)
                const float wj = p.general ? (cb ? sm.tw : S.gw)[jv] : beta;
                const float uu = (p.erase || p.general) ? __fsub_rn(__fmul_rn(wj, vj), P) : vj;
                sm.u[jv] = uu;
                p.o[tok * DV + jv] = fmaf(uu, kq, Rr);
            } else if (prep_k && t + 1 < p.t_end) {
                // the next token's inputs into buffer cb ^ 1, whose contents (the previous
                // token's) were last read before the previous B4.  k goes to the third k
                // buffer: this token's k is read after the coming B4, the previous token's was
                // last read before this token's B3.
                const int i = pi, nb = cb ^ 1, nk3 = k3 == 2 ? 0 : k3 + 1;
                const float nbeta = rbeta, nk = rk, nq = rq;
                float rate;
                if (p.s_code) {
                    const int code = min(rc, p.L - 1);
                    if (p.decay_row)
                        rate = p.L <= 4 ? S.lut[i * p.L + code]
                                        : __ldg(p.s_lut + (static_cast<size_t>(h) * DK + i) * p.L + code);
                    else
                        rate = __ldg(p.s_lut + static_cast<size_t>(h) * p.L + code);
                } else {
                    rate = rs;
                }
                if (!(rate > 0.0f) || !(rate < INFINITY)) raise_status(p.status, QS_DEV_RATE);
                (nk3 == 0 ? S.k : nk3 == 1 ? sm.tk : sm.tk2)[i] = nk;
                (nb ? sm.tq : S.q)[i] = nq;
                (nb ? sm.d1 : sm.d)[i] = expf(-rate);
                (nb ? sm.a1 : sm.a)[i] = p.general ? ra : __fmul_rn(nbeta, nk);
                if (prep_v) {
                    (nb ? sm.tv : S.v)[i] = rv;
                    if (p.general) (nb ? sm.tw : S.gw)[i] = rw;
                }
                if (i == 0) sm.tbeta[nb] = nbeta;
                if (stats) {
                    const float xs = -expm1f(-2.0f * rate);
                    if (p.general) {
                        sm.rowR[i] = xs;   // the erasure term needs all of the next k: after B4
                    } else {
                        const float xr = p.erase ? __fmul_rn(__fmul_rn(nbeta, __fsub_rn(2.0f, nbeta)), __fmul_rn(nk, nk)) : 0.0f;
                        S.ms[i] = __fadd_rn(S.ms[i], __fmul_rn(p.alpha, __fsub_rn(xs, S.ms[i])));
                        S.mr[i] = __fadd_rn(S.mr[i], __fmul_rn(p.alpha, __fsub_rn(xr, S.mr[i])));
                    }
                }
                const float s2 = warp_sum(nk * nq);
                if (lane == 0) sm.wsum[nb][i >> 5] = s2;
                if (t + 2 < p.t_end) load_raw(tok + 2 * static_cast<size_t>(p.H));
            }
            __syncthreads();                                                           // B4
            if (prep_k && t + 1 < p.t_end && p.general && stats) {
                // the general erasure statistic of the next token (needs all of its k)
                const int nk3 = k3 == 2 ? 0 : k3 + 1;
                const float* kb = nk3 == 0 ? S.k : nk3 == 1 ? sm.tk : sm.tk2;
                const float xr = general_erasure<DK>((cb ? sm.a : sm.a1)[pi], kb[pi], kb);
                S.ms[pi] = __fadd_rn(S.ms[pi], __fmul_rn(p.alpha, __fsub_rn(sm.rowR[pi], S.ms[pi])));
                S.mr[pi] = __fadd_rn(S.mr[pi], __fmul_rn(p.alpha, __fsub_rn(xr, S.mr[pi])));
            }
            if constexpr (RS == 2) {
                const float2 u0 = reinterpret_cast<const float2*>(&sm.u[cl * 4])[0];
                const float2 u1 = reinterpret_cast<const float2*>(&sm.u[cl * 4])[1];
#pragma unroll
                for (int jr = 0; jr < NSL; ++jr) {
                    const float kk = kv[warp * RPW + jr * RS + half];
                    x[jr][0] = __ffma2_rn(make_float2(kk, kk), u0, x[jr][0]);
                    x[jr][1] = __ffma2_rn(make_float2(kk, kk), u1, x[jr][1]);
                }
            } else {
            float2 u2[CP2];
#pragma unroll
            for (int c = 0; c < CP2; ++c) u2[c] = reinterpret_cast<const float2*>(&sm.u[lane * CPL])[c];
#pragma unroll
            for (int r4 = 0; r4 < RPW; r4 += 4) {
                const float4 k4 = *reinterpret_cast<const float4*>(&kv[warp * RPW + r4]);
                const float ks[4] = {k4.x, k4.y, k4.z, k4.w};
#pragma unroll
                for (int j4 = 0; j4 < 4; ++j4) {
                    const float2 k2 = make_float2(ks[j4], ks[j4]);
#pragma unroll
                    for (int c = 0; c < CP2; ++c) x[r4 + j4][c] = __ffma2_rn(k2, u2[c], x[r4 + j4][c]);
                }
            }
            }
        }

        // the payload buffer is free: the next head's packed rows
        if (has_next) wb_issue_payload<DK, DV>(sm.st[sidx ^ 1], pay, g + 1, wp);
        // state to the buffer
#pragma unroll
        for (int r = 0; r < NSL; ++r) {
            const int i = warp * RPW + r * RS + half;
            *reinterpret_cast<float4*>(sm.sbuf + sb_off<DV>(i, cl)) =
                make_float4(x[r][0].x, x[r][0].y, x[r][1].x, x[r][1].y);
        }
        if constexpr (CHUNK) {
            __syncthreads();
            chunk_interval(p, S, sm.sbuf, cb, tmem, mphase, b, h, stats);
        }
        __syncthreads();                                                               // B5

        // ---- write-back (row layout) ----------------------------------------------------------
        const bool refit = (p.fit_every <= 1) || ((p.w_index + h) % p.fit_every == 0);
        // Row batches are claimed dynamically (longest first, by the order above): the
        // search length varies with the width and the data.
        auto next_batch = [&]() {
            int nb = 0;
            if (lane == 0) nb = atomicAdd(&sm.bat_next, 1);
            return __shfl_sync(kFull, nb, 0);
        };
        for (int bat = warp; bat < NB; bat = next_batch()) {
            const int i = sm.ord_out[bat * RPB + lane / TPR], q = lane % TPR;
            const int w = S.w_out[i];
            float2 xv[16], av[16];
#pragma unroll
            for (int g2 = 0; g2 < 8; ++g2) {
                const float4 v = *reinterpret_cast<const float4*>(sm.sbuf + sb_off<DV>(i, 8 * q + g2));
                xv[2 * g2] = make_float2(v.x, v.y);
                xv[2 * g2 + 1] = make_float2(v.z, v.w);
            }
            // row range R = max |x| (identical in the row's TPR lanes)
            float m4[4] = {0.0f, 0.0f, 0.0f, 0.0f};
#pragma unroll
            for (int c = 0; c < 16; ++c) {
                av[c] = make_float2(fabsf(xv[c].x), fabsf(xv[c].y));
                m4[c & 3] = fmaxf(m4[c & 3], fmaxf(av[c].x, av[c].y));
            }
            const float lmax = fmaxf(fmaxf(m4[0], m4[1]), fmaxf(m4[2], m4[3]));
            float R = lmax;
#pragma unroll
            for (int o = 1; o < TPR; o <<= 1) R = fmaxf(R, __shfl_xor_sync(kFull, R, o));
            if (p.mode == 1) {   // statistics only: the range is all this pass produces
                if (q == 0) sm.rowR[i] = R;
                continue;
            }
            float D = 0.0f;
            int fidx = S.fidx[i];
            if (__any_sync(kFull, w == 1)) {
                // 1-bit rows: mean |x|
                float2 s2 = make_float2(0.0f, 0.0f);
#pragma unroll
                for (int c = 0; c < 16; ++c) s2 = __fadd2_rn(s2, av[c]);
                float sum = s2.x + s2.y;
#pragma unroll
                for (int o = 1; o < TPR; o <<= 1) sum += __shfl_xor_sync(kFull, sum, o);
                if (w == 1) D = f16_round(__fdiv_rn(sum, static_cast<float>(DV)));
            }
            const float inv_n = sm.wc[w > 16 ? 0 : w].y;
            if (refit) {
                __syncwarp();   // the previous batch's rows are done with the candidate table
                // the row's 16 candidate steps, KPT per lane.  The search takes approximate
                // reciprocals; the chosen step's IEEE reciprocal is taken below for the codes.
#pragma unroll
                for (int kk = 0; kk < KPT; ++kk) {
                    const int k = q * KPT + kk;
                    const float Dk = (w >= 2 && R > 0.0f) ? cand_step(sm.fitf[k], R, inv_n) : 0.0f;
                    float ik = 0.0f;
                    if (Dk > 0.0f) asm("rcp.approx.ftz.f32 %0, %1;" : "=f"(ik) : "f"(Dk));
                    sm.rc.cand[warp][lane / TPR][k] = make_float2(ik, -Dk);
                }
                __syncwarp();
                // squared error of the candidates (levels clamped at n): e = |x| - q Delta,
                // q = min(rint(|x| / Delta), n); the smallest wins, ties to the larger factor.
                // Candidates are taken from the largest factor down, two per round (independent
                // work for the warp).  Every element at or above n Delta_k quantises to n, so the
                // clipping error of the lanes' maxima is a lower bound on candidate k's error that
                // grows as k falls: once it exceeds the best error found (with a 2^-10 margin for
                // rounding), no smaller factor can win.  The round's second candidate is evaluated
                // even when its bound already rules it out; it then cannot win the comparison.
                const float lim = sm.wc[w > 16 ? 0 : w].w, nf = sm.wc[w > 16 ? 0 : w].x;
                float mx[TPR];
#pragma unroll
                for (int jl = 0; jl < TPR; ++jl) mx[jl] = __shfl_sync(kFull, lmax, (lane & ~(TPR - 1)) + jl);
                const float2 M2 = make_float2(kMagic, kMagic), nM2 = make_float2(-kMagic, -kMagic);
                const float2* crow = sm.rc.cand[warp][lane / TPR];
                float bsse = INFINITY;
                int bk = kNFit - 1;
                // each round's two candidates are loaded one round ahead
                float2 pA = crow[kNFit - 1], pB = crow[kNFit - 2];
#pragma unroll 1
                for (int k = kNFit - 1; k >= 0; k -= 2) {
                    // candidates k and k - 1 in one round (k - 1 may not exist)
                    const bool two = k >= 1;
                    const float2 cA = pA, cB = two ? pB : pA;
                    if (k >= 3) {
                        pA = crow[k - 2];
                        pB = crow[k - 3];
                    }
                    const float LA = -nf * cA.y, LB = -nf * cB.y;
                    float lbA = 0.0f;
#pragma unroll
                    for (int jl = 0; jl < TPR; ++jl) {
                        const float e = fmaxf(mx[jl] - LA, 0.0f);
                        lbA = fmaf(e, e, lbA);
                    }
                    const bool goA = w >= 2 && lbA <= bsse * (1.0f + 1.0f / 1024.0f);
                    if (!__any_sync(kFull, goA)) break;
                    const float2 iA = make_float2(cA.x, cA.x), dA = make_float2(cA.y, cA.y);
                    const float2 iB = make_float2(cB.x, cB.x), dB = make_float2(cB.y, cB.y);
                    float2 aA0 = make_float2(0.0f, 0.0f), aA1 = aA0, aB0 = aA0, aB1 = aA0;
#pragma unroll
                    for (int c = 0; c < 16; c += 2) {
                        float2 t0 = __ffma2_rn(av[c], iA, M2);
                        float2 t1 = __ffma2_rn(av[c + 1], iA, M2);
                        float2 u0 = __ffma2_rn(av[c], iB, M2);
                        float2 u1 = __ffma2_rn(av[c + 1], iB, M2);
                        t0.x = fminf(t0.x, lim); t0.y = fminf(t0.y, lim);
                        t1.x = fminf(t1.x, lim); t1.y = fminf(t1.y, lim);
                        u0.x = fminf(u0.x, lim); u0.y = fminf(u0.y, lim);
                        u1.x = fminf(u1.x, lim); u1.y = fminf(u1.y, lim);
                        const float2 e0 = __ffma2_rn(__fadd2_rn(t0, nM2), dA, av[c]);
                        const float2 e1 = __ffma2_rn(__fadd2_rn(t1, nM2), dA, av[c + 1]);
                        const float2 f0 = __ffma2_rn(__fadd2_rn(u0, nM2), dB, av[c]);
                        const float2 f1 = __ffma2_rn(__fadd2_rn(u1, nM2), dB, av[c + 1]);
                        aA0 = __ffma2_rn(e0, e0, aA0);
                        aA1 = __ffma2_rn(e1, e1, aA1);
                        aB0 = __ffma2_rn(f0, f0, aB0);
                        aB1 = __ffma2_rn(f1, f1, aB1);
                    }
                    float tA = (aA0.x + aA0.y) + (aA1.x + aA1.y);
                    float tB = (aB0.x + aB0.y) + (aB1.x + aB1.y);
#pragma unroll
                    for (int o = 1; o < TPR; o <<= 1) {
                        tA += __shfl_xor_sync(kFull, tA, o);
                        tB += __shfl_xor_sync(kFull, tB, o);
                    }
                    if (goA && tA < bsse) {
                        bsse = tA;
                        bk = k;
                    }
                    if (two && w >= 2 && tB < bsse) {
                        bsse = tB;
                        bk = k - 1;
                    }
                }
                if (w >= 2) {
                    D = -sm.rc.cand[warp][lane / TPR][bk].y;
                    fidx = bk;
                }
            } else if (w >= 2 && R > 0.0f) {
                D = cand_step(sm.fitf[fidx], R, inv_n);
            }
            if (q == 0) {
                sm.rowR[i] = R;
                sm.out_scale[i] = f16_bits(D);
                sm.out_fidx[i] = static_cast<uint8_t>(fidx);
            }
            // codes + packed words, stored to the output region (4w bytes at byte 4 w q of the row)
            uint8_t* orow = p.out_payload + static_cast<size_t>(b) * p.region_bytes + S.out_off + sm.off_out[i];
            pack_row<DV == 128 ? 16 : 8>(w, xv, w >= 2 ? step_rcp(D) : 0.0f, orow + 4 * w * q);
        }
        __syncthreads();                                                               // B6
        // ---- stores -------------------------------------------------------------------------------
        const size_t rb = static_cast<size_t>(g) * DK;
        if (tid < DK) {
            if (p.mode != 1) {
                p.out_scales[rb + tid] = sm.out_scale[tid];
                p.out_fidx[rb + tid] = sm.out_fidx[tid];
            }
            if (p.range) p.range[rb + tid] = sm.rowR[tid];
            if (stats && p.mode != 2) {
                p.ema_s[rb + tid] = S.ms[tid];
                p.ema_r[rb + tid] = S.mr[tid];
            }
        }
    }
    if constexpr (CHUNK) chunk_teardown(tmem, cb, p.status);
}

template <int DK, int DV, int NW, bool CHUNK = false>
cudaError_t launch_wb_row_t(const qstate_cfg& cfg, const StepParams& sp, cudaStream_t stream) {
    auto kern = wb_row_kernel<DK, DV, NW, CHUNK>;
    WbParams wp;
    wp.s = sp;
    wp.s.stage_bytes = DK * DV * cfg.bmax / 8;
    wp.nheads = cfg.B * cfg.H;
    const int pstride = (wp.s.stage_bytes + 32 + 15) & ~15;
    const size_t smem = sizeof(WbSmem<DK, DV, NW>) + static_cast<size_t>(pstride) + (CHUNK ? ChunkGeo::kBytes : 0u);
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
