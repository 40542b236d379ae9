// qs_alloc.cu -- bit allocation (Sec. 3 "State bit allocation": Eq. 3, Eq. 4 and the integer
// rounding to the layer budget), one CTA of 1024 threads per batch element.
//
// Weights c_i = Gamma_hat_i Rtilde_i^2 are formed in FP32 with one IEEE rounding per operation
// (Gamma_hat = (1 - m_s) / (expm1(m_r) + m_s), expm1 from its Taylor series), so they are
// reproducible bit for bit.  Rounding Eq. (4) to nearest, clipping and adjusting to the budget
// by the rounding remainders hands out bits in decreasing order of their marginal value
// c_i 4^{-b}: the result is the set of the M = total - N b_min most valuable bits (i, b),
// b in (b_min, b_max].  For FP32 c the order of c 4^{-b} is the order of the integer key
// bits(c) - b 2^24 (a power-of-4 scaling moves only the exponent field), so the kernel finds
// the M-th largest key from integer counts -- no logarithm, no floating-point
// comparison -- and gives bits tied at the threshold to the lowest unit indices.  The M-th
// largest key is found from a histogram of the keys' high parts followed by a radix select on
// their low 24 bits.
#include "qs_common.cuh"

namespace qs {

namespace {

constexpr int kThreads = 1024;
constexpr int kNullKey = -73 * (1 << 23);   // bits of 2^-200 on a virtual exponent
constexpr int kHistOff = 64;                 // high parts -37 - 16 .. 127 -> bins 11 .. 191

__device__ __forceinline__ float expm1_series(float x, const float* e1) {
    if (!(x > 0.0f)) return 0.0f;
    int halvings = 0;
    while (x > 1.0f) {
        x = __fmul_rn(x, 0.5f);
        ++halvings;
    }
    float p = e1[16];
#pragma unroll
    for (int k = 15; k >= 1; --k) p = __fadd_rn(__fmul_rn(p, x), e1[k]);
    float y = __fmul_rn(p, x);
    for (int i = 0; i < halvings; ++i) y = __fmul_rn(y, __fadd_rn(y, 2.0f));
    return y;
}

// Exclusive prefix sum over the block of one int per thread (thread order).
__device__ int block_exclusive_scan(int v, int* red, int* total) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    int incl = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        int n = __shfl_up_sync(kFull, incl, o);
        if (lane >= o) incl += n;
    }
    __syncthreads();
    if (lane == 31) red[warp] = incl;
    __syncthreads();
    if (warp == 0) {
        int w = red[lane];
        int wi = w;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            int n = __shfl_up_sync(kFull, wi, o);
            if (lane >= o) wi += n;
        }
        red[32 + lane] = wi - w;
        if (lane == 31) red[64] = wi;
    }
    __syncthreads();
    const int r = red[32 + warp] + incl - v;
    *total = red[64];
    return r;
}

}  // namespace

// Group of unit u: a shift when the group size gsz is a power of two (gshift >= 0), else a
// division.
__device__ __forceinline__ int group_of(int u, int gsz, int gshift) { return gshift >= 0 ? u >> gshift : u / gsz; }

// Allocation weight c_u (Eq. 3 and the alternatives of Table 1), one IEEE rounding per
// operation.  ms_s / mr_s: the batch element's EMA statistics; Rs / gmean: its ranges, stored
// with one padding word after every group of gsz units, and the group means of R^2 (row unit).
__device__ float weight(const AllocParams& p, int u, const float* ms_s, const float* mr_s, const float* Rs,
                        const float* gmean, int gsz, int gshift) {
    const int kind = p.weight_kind;
    float R2 = 1.0f, rt2 = 1.0f;   // R^2 and Rtilde^2 (1 for the head unit)
    if (p.unit_row) {
        const int gi = group_of(u, gsz, gshift);
        const float R = Rs[u + gi];
        R2 = __fmul_rn(R, R);
        const float m = gmean[gi];
        if (m > 0.0f) rt2 = __fdiv_rn(R2, m);
    }
    if (kind == QSTATE_WEIGHT_RANGE) return R2;
    if (kind == QSTATE_WEIGHT_NRANGE) return rt2;
    // statistics of the unit itself, or of unit pi(u) for the shuffled decay weights
    const int us = kind == QSTATE_WEIGHT_SHUFFLE
                       ? static_cast<int>((static_cast<long long>(p.shuf_a) * u + p.shuf_b) % p.units)
                       : u;
    const float ms = ms_s[us];
    if (kind == QSTATE_WEIGHT_PERSIST) return __fmul_rn(__fdiv_rn(1.0f, ms), rt2);
    if (kind == QSTATE_WEIGHT_WBFACTOR) {
        float pw = 1.0f, bb = __fsub_rn(1.0f, ms);   // (1 - m_s)^C, low bit first
        for (int e = p.C; e > 0; e >>= 1) {
            if (e & 1) pw = __fmul_rn(pw, bb);
            bb = __fmul_rn(bb, bb);
        }
        return __fmul_rn(__fdiv_rn(1.0f, __fsub_rn(1.0f, pw)), rt2);
    }
    float mr = kind == QSTATE_WEIGHT_NOERASE ? 0.0f : mr_s[us];
    if (mr < 0.0f) mr = 0.0f;
    const float G = __fdiv_rn(__fsub_rn(1.0f, ms), __fadd_rn(expm1_series(mr, p.e1), ms));
    if (kind == QSTATE_WEIGHT_GAMMA_RAW) return __fmul_rn(G, R2);
    return __fmul_rn(G, rt2);   // OURS, NOERASE, SHUFFLE
}

// Warp 0 only: the bin whose suffix count (bins >= it, highest first) first reaches `rank`
// (1-based); returns it and sets *above to the count of the bins above it.  hist has 256 bins.
__device__ int warp_select_bin(const int* hist, int rank, int* above) {
    const int lane = threadIdx.x & 31;
    // lane l owns bins [8 (31 - l), 8 (31 - l) + 8): lanes in descending bin order
    int c[8];
    int s = 0;
#pragma unroll
    for (int k = 0; k < 8; ++k) {
        c[k] = hist[8 * (31 - lane) + 7 - k];   // descending within the lane
        s += c[k];
    }
    int incl = s;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const int n = __shfl_up_sync(kFull, incl, o);
        if (lane >= o) incl += n;
    }
    const int excl = incl - s;   // count of all bins above this lane's
    const unsigned hit = __ballot_sync(kFull, excl < rank && incl >= rank);
    const int src = __ffs(hit) - 1;
    int bin = 0, ab = 0;
    if (lane == src) {
        int run = excl;
#pragma unroll
        for (int k = 0; k < 8; ++k) {
            if (run + c[k] >= rank) {
                bin = 8 * (31 - lane) + 7 - k;
                ab = run;
                break;
            }
            run += c[k];
        }
    }
    bin = __shfl_sync(kFull, bin, src);
    *above = __shfl_sync(kFull, ab, src);
    return bin;
}

__global__ void __launch_bounds__(kThreads, 2) alloc_kernel(const AllocParams p) {
    extern __shared__ __align__(16) uint8_t smem[];
    const int N = p.units;
    int* key = reinterpret_cast<int*>(smem);
    const int gsz = p.group_heads * p.dk;
    const int gshift = (gsz & (gsz - 1)) == 0 ? __ffs(gsz) - 1 : -1;
    const int ngroups = p.unit_row ? N / gsz : 0;
    // the EMA statistics are read once each, from global memory (the write-back just wrote
    // them: L2); only the ranges, read twice, are staged
    const size_t base = static_cast<size_t>(blockIdx.x) * N;
    const float* ms_s = p.uniform ? nullptr : p.ema_s + base;
    const float* mr_s = p.uniform ? nullptr : p.ema_r + base;
    float* Rs = reinterpret_cast<float*>(key + N);                     // row unit: ranges, a padding
                                                                       // word after each group
    float* gmean = Rs + (p.unit_row ? N + ngroups : 0);
    int* hist = reinterpret_cast<int*>(gmean + ((ngroups + 3) & ~3));
    int* redi = hist + 1024;                                           // hist: 256 bins, then H head sizes
    int* sel = redi + 72;                                              // H*, rank, low prefix
    uint8_t* wv = reinterpret_cast<uint8_t*>(sel + 4);
    const int tid = threadIdx.x;

    // 1. ranges staged in shared memory (row unit; independent coalesced loads); mean R^2 of
    //    each output-normalisation group, summed in row order.  Group g's ranges sit at stride
    //    gsz + 1, so the threads summing different groups in lockstep hit different banks.
    if (!p.uniform) {
        if (p.unit_row)
            for (int u = tid; u < N; u += kThreads) Rs[u + group_of(u, gsz, gshift)] = p.range[base + u];
        __syncthreads();
        if (p.unit_row) {
            // one thread per group, its sum a chain of gsz dependent additions: the next 16
            // ranges are loaded while the current 16 are added
            for (int g = tid; g < ngroups; g += kThreads) {
                const float* rg = Rs + g * (gsz + 1);
                float acc = 0.0f;
                constexpr int PF = 16;
                float cur[PF];
                const int full = gsz - gsz % PF;
#pragma unroll
                for (int k = 0; k < PF; ++k) cur[k] = k < gsz ? rg[k] : 0.0f;
                for (int r = 0; r < full; r += PF) {
                    float nxt[PF];
#pragma unroll
                    for (int k = 0; k < PF; ++k) nxt[k] = r + PF + k < gsz ? rg[r + PF + k] : 0.0f;
#pragma unroll
                    for (int k = 0; k < PF; ++k) acc = __fadd_rn(acc, __fmul_rn(cur[k], cur[k]));
#pragma unroll
                    for (int k = 0; k < PF; ++k) cur[k] = nxt[k];
                }
                for (int r = full; r < gsz; ++r) acc = __fadd_rn(acc, __fmul_rn(rg[r], rg[r]));
                gmean[g] = __fdiv_rn(acc, static_cast<float>(gsz));
            }
        }
    }
    for (int k = tid; k < 256; k += kThreads) hist[k] = 0;
    __syncthreads();

    // 2. weights (Eq. 3) -> integer keys; the keys of unit u's bits b_min + j (j = 1..J) are
    //    key_u - j 2^24, i.e. high part (key_u >> 24) - j and low part key_u & 0xFFFFFF, so every
    //    unit adds one to a contiguous range of high parts: a difference array on 256 bins
    const int J = p.bmax - p.bmin;
    const long long M = p.total - static_cast<long long>(N) * p.bmin;
    for (int u = tid; u < N; u += kThreads) {
        float c = 1.0f;
        if (!p.uniform) c = weight(p, u, ms_s, mr_s, Rs, gmean, gsz, gshift);
        if (c > 0x1p60f) c = 0x1p60f;
        const int k = (c >= 0x1p-60f) ? __float_as_int(c) : kNullKey;
        key[u] = k;
    }
    // lanes with equal high parts add together (one atomic per distinct value and warp)
    if (J > 0) {
        for (int u0w = tid - (tid & 31); u0w < N; u0w += kThreads) {
            const int u = u0w + (tid & 31);
            const bool in = u < N;
            const int E = in ? (key[u] >> 24) : 0x7fffffff;   // in [-37, 127]
            const unsigned peers = __match_any_sync(kFull, E);
            if (in && (tid & 31) == __ffs(peers) - 1) {
                const int cnt = __popc(peers);
                atomicAdd(&hist[E - J + kHistOff], cnt);
                atomicAdd(&hist[E + kHistOff], -cnt);
            }
        }
    }
    __syncthreads();

    // 3. V = the M-th largest key: its high part from the bins (prefix of the difference
    //    array), then its low 24 bits by a radix select (8 bits per pass) over the units whose
    //    key range covers that high part
    long long V = LLONG_MAX;   // M == 0: nothing above b_min
    if (M > 0) {
        if (tid < 32) {
            // prefix sum over 256 bins -> counts per high part
            int c[8];
            int s = 0;
#pragma unroll
            for (int k = 0; k < 8; ++k) {
                s += hist[8 * tid + k];
                c[k] = s;
            }
            int incl = s;
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                const int n = __shfl_up_sync(kFull, incl, o);
                if (tid >= o) incl += n;
            }
            const int ex = incl - s;
            __syncwarp();
#pragma unroll
            for (int k = 0; k < 8; ++k) hist[8 * tid + k] = ex + c[k];
            __syncwarp();
            int above = 0;
            const int hb = warp_select_bin(hist, static_cast<int>(M), &above);
            if (tid == 0) {
                sel[0] = hb - kHistOff;                  // high part of V
                sel[1] = static_cast<int>(M) - above;    // rank of V among that bin's keys
                sel[2] = 0;                              // low bits found so far
            }
        }
        __syncthreads();
        const int Hs = sel[0];
#pragma unroll 1
        for (int pass = 0; pass < 3; ++pass) {
            const int sh = 16 - 8 * pass;
            const int pre = sel[2];
            const int pmask = pass == 0 ? 0 : (0xFFFFFF << (sh + 8)) & 0xFFFFFF;
            for (int k = tid; k < 256; k += kThreads) hist[k] = 0;
            __syncthreads();
            for (int u = tid; u < N; u += kThreads) {
                const int k = key[u];
                const int E = k >> 24, L = k & 0xFFFFFF;
                if (E - J <= Hs && Hs <= E - 1 && (L & pmask) == pre) atomicAdd(&hist[(L >> sh) & 255], 1);
            }
            __syncthreads();
            if (tid < 32) {
                int above = 0;
                const int d = warp_select_bin(hist, sel[1], &above);
                if (tid == 0) {
                    sel[1] -= above;
                    sel[2] = pre | (d << sh);
                }
            }
            __syncthreads();
        }
        V = static_cast<long long>(Hs) * (1LL << 24) + sel[2];
    }

    // 4. widths: bits strictly above V, plus tied bits to the lowest unit indices
    const int per = (N + kThreads - 1) / kThreads;
    const int u0 = tid * per, u1 = min(N, u0 + per);
    int gt_local = 0, tie_local = 0;
    for (int u = u0; u < u1; ++u) {
        int gt = 0, tie = 0;
        if (M > 0) {
            const long long d = static_cast<long long>(key[u]) - V;
            if (d > 0) {
                gt = static_cast<int>(min((d - 1) >> 24, static_cast<long long>(J)));
                tie = ((d & 0xFFFFFF) == 0 && (d >> 24) <= J) ? 1 : 0;
            }
        }
        wv[u] = static_cast<uint8_t>(p.bmin + gt);
        gt_local += gt;
        tie_local += tie;
    }
    int gt_total = 0;
    (void)block_exclusive_scan(gt_local, redi, &gt_total);
    const long long need = M - gt_total;
    int tie_total = 0;
    int tie_before = block_exclusive_scan(tie_local, redi, &tie_total);
    for (int u = u0; u < u1; ++u) {
        if (M > 0) {
            const long long d = static_cast<long long>(key[u]) - V;
            if (d > 0 && (d & 0xFFFFFF) == 0 && (d >> 24) <= J) {
                if (tie_before < need) wv[u] += 1;
                ++tie_before;
            }
        }
        p.widths[base + u] = wv[u];
    }
    __syncthreads();

    // 5. head offsets: exclusive prefix sum of the heads' payload bytes (row unit: one warp
    //    per head sums its widths)
    int* hbytes = hist;   // free again
    if (p.unit_row) {
        for (int h = tid >> 5; h < p.H; h += kThreads / 32) {
            int sum = 0;
            for (int i = tid & 31; i < p.dk; i += 32) sum += wv[h * p.dk + i];
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) sum += __shfl_xor_sync(kFull, sum, o);
            if ((tid & 31) == 0) hbytes[h] = sum * (p.dv / 8);
        }
    } else {
        for (int h = tid; h < p.H; h += kThreads) hbytes[h] = wv[h] * p.dk * p.dv / 8;
    }
    __syncthreads();
    int total_bytes = 0;
    const int off = block_exclusive_scan(tid < p.H ? hbytes[tid] : 0, redi, &total_bytes);
    if (tid < p.H) p.head_off[static_cast<size_t>(blockIdx.x) * p.H + tid] = static_cast<uint32_t>(off);
    if (tid == 0 && M > 0 && (need < 1 || need > tie_total)) raise_status(p.status, QS_DEV_LAYOUT);
}

cudaError_t launch_alloc(const AllocParams& p, cudaStream_t stream) {
    const int ngroups = p.unit_row ? p.units / (p.group_heads * p.dk) : 0;
    const size_t smem = static_cast<size_t>(p.units) * 4 + (p.unit_row ? (p.units + ngroups) * 4 : 0) +
                        ((ngroups + 3) & ~3) * 4 + 1024 * 4 + 72 * 4 + 4 * 4 + p.units + 16;
    cudaError_t e = cudaFuncSetAttribute(alloc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         static_cast<int>(smem));
    if (e != cudaSuccess) return e;
    alloc_kernel<<<p.B, kThreads, smem, stream>>>(p);
    return cudaGetLastError();
}

}  // namespace qs
