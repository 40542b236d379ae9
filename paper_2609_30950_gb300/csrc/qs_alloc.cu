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
// the M-th largest key by bisection on integer counts -- no logarithm, no floating-point
// comparison -- and gives bits tied at the threshold to the lowest unit indices.
#include "qs_common.cuh"

namespace qs {

namespace {

constexpr int kThreads = 1024;
constexpr long long kNullKey = -73LL * (1LL << 23);   // bits of 2^-200 on a virtual exponent

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

template <typename T>
__device__ T block_reduce(T v, T* red, int op) {   // op 0: sum, 1: min, 2: max
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        T w = __shfl_xor_sync(kFull, v, o);
        v = op == 0 ? v + w : (op == 1 ? (w < v ? w : v) : (w > v ? w : v));
    }
    __syncthreads();
    if (lane == 0) red[warp] = v;
    __syncthreads();
    if (warp == 0) {
        v = red[lane];   // blockDim.x == 1024: 32 warps
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
            T w = __shfl_xor_sync(kFull, v, o);
            v = op == 0 ? v + w : (op == 1 ? (w < v ? w : v) : (w > v ? w : v));
        }
        if (lane == 0) red[0] = v;
    }
    __syncthreads();
    T r = red[0];
    return r;
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

__global__ void __launch_bounds__(kThreads) alloc_kernel(const AllocParams p) {
    extern __shared__ __align__(16) uint8_t smem[];
    const int N = p.units;
    long long* key = reinterpret_cast<long long*>(smem);
    const int gsz = p.group_heads * p.dk;
    const int ngroups = p.unit_row ? N / gsz : 0;
    float* Rs = reinterpret_cast<float*>(key + N);                   // row unit: ranges
    float* gmean = Rs + (p.unit_row ? N : 0);
    long long* redl = reinterpret_cast<long long*>(gmean + ((ngroups + 3) & ~3));
    int* redi = reinterpret_cast<int*>(redl + 32);
    uint8_t* wv = reinterpret_cast<uint8_t*>(redi + 72);
    const int tid = threadIdx.x;
    const size_t base = static_cast<size_t>(blockIdx.x) * N;

    // 1. mean R^2 of each output-normalisation group, summed in row order (row unit); the
    //    ranges are staged in shared memory first so the sequential sums read on-chip data
    if (!p.uniform && p.unit_row) {
        for (int u = tid; u < N; u += kThreads) Rs[u] = p.range[base + u];
        __syncthreads();
        for (int g = tid; g < ngroups; g += kThreads) {
            float acc = 0.0f;
#pragma unroll 8
            for (int r = g * gsz; r < (g + 1) * gsz; ++r) acc = __fadd_rn(acc, __fmul_rn(Rs[r], Rs[r]));
            gmean[g] = __fdiv_rn(acc, static_cast<float>(gsz));
        }
    }
    __syncthreads();

    // 2. weights (Eq. 3) -> integer keys
    long long kmin = LLONG_MAX, kmax = LLONG_MIN;
    for (int u = tid; u < N; u += kThreads) {
        float c = 1.0f;
        if (!p.uniform) {
            const float ms = p.ema_s[base + u];
            float mr = p.ema_r[base + u];
            if (mr < 0.0f) mr = 0.0f;
            const float G = __fdiv_rn(__fsub_rn(1.0f, ms), __fadd_rn(expm1_series(mr, p.e1), ms));
            float rt2 = 1.0f;
            if (p.unit_row) {
                const float m = gmean[u / gsz];
                const float R = Rs[u];
                if (m > 0.0f) rt2 = __fdiv_rn(__fmul_rn(R, R), m);
            }
            c = __fmul_rn(G, rt2);
        }
        if (c > 0x1p60f) c = 0x1p60f;
        const long long k = (c >= 0x1p-60f) ? static_cast<long long>(__float_as_int(c)) : kNullKey;
        key[u] = k;
        kmin = k < kmin ? k : kmin;
        kmax = k > kmax ? k : kmax;
    }
    kmin = block_reduce<long long>(kmin, redl, 1);
    kmax = block_reduce<long long>(kmax, redl, 2);

    // 3. the M-th most valuable bit: largest T with #{(u, j): key_u - j 2^24 >= T} >= M
    const int J = p.bmax - p.bmin;
    const long long M = p.total - static_cast<long long>(N) * p.bmin;
    long long V = LLONG_MAX;   // M == 0: nothing above b_min
    if (M > 0) {
        long long lo = kmin - static_cast<long long>(J) * (1LL << 24);   // count(lo) = N J >= M
        long long hi = kmax - (1LL << 24) + 1;                          // count(hi) = 0 < M
        while (hi - lo > 1) {
            const long long mid = lo + (hi - lo) / 2;
            int cnt = 0;
            for (int u = tid; u < N; u += kThreads) {
                const long long d = key[u] - mid;
                if (d >= 0) cnt += static_cast<int>(min(d >> 24, static_cast<long long>(J)));
            }
            cnt = block_reduce<int>(cnt, redi, 0);
            if (cnt >= M) lo = mid; else hi = mid;
        }
        V = lo;
    }

    // 4. widths: bits strictly above V, plus tied bits to the lowest unit indices
    const int per = (N + kThreads - 1) / kThreads;
    const int u0 = tid * per, u1 = min(N, u0 + per);
    int gt_local = 0, tie_local = 0;
    for (int u = u0; u < u1; ++u) {
        int gt = 0, tie = 0;
        if (M > 0) {
            const long long d = key[u] - V;
            if (d > 0) {
                gt = static_cast<int>(min((d - 1) >> 24, static_cast<long long>(J)));
                tie = ((d & 0xFFFFFF) == 0 && (d >> 24) <= J) ? 1 : 0;
            }
        }
        wv[u] = static_cast<uint8_t>(p.bmin + gt);
        gt_local += gt;
        tie_local += tie;
    }
    const int gt_total = block_reduce<int>(gt_local, redi, 0);
    const long long need = M - gt_total;
    int tie_total = 0;
    int tie_before = block_exclusive_scan(tie_local, redi, &tie_total);
    for (int u = u0; u < u1; ++u) {
        if (M > 0) {
            const long long d = key[u] - V;
            if (d > 0 && (d & 0xFFFFFF) == 0 && (d >> 24) <= J) {
                if (tie_before < need) wv[u] += 1;
                ++tie_before;
            }
        }
        p.widths[base + u] = wv[u];
    }
    __syncthreads();

    // 5. head offsets: exclusive prefix sum of the heads' payload bytes
    int hb = 0;
    for (int h = tid; h < p.H; h += kThreads) {   // H <= 1024 (validated)
        if (p.unit_row) {
            for (int i = 0; i < p.dk; ++i) hb += wv[h * p.dk + i];
            hb *= p.dv / 8;
        } else {
            hb = wv[h] * p.dk * p.dv / 8;
        }
    }
    int total_bytes = 0;
    const int off = block_exclusive_scan(tid < p.H ? hb : 0, redi, &total_bytes);
    if (tid < p.H) p.head_off[static_cast<size_t>(blockIdx.x) * p.H + tid] = static_cast<uint32_t>(off);
    if (tid == 0 && (need < 0 || need > tie_total)) raise_status(p.status, QS_DEV_LAYOUT);
}

cudaError_t launch_alloc(const AllocParams& p, cudaStream_t stream) {
    const int ngroups = p.unit_row ? p.units / (p.group_heads * p.dk) : 0;
    const size_t smem = static_cast<size_t>(p.units) * 8 + (p.unit_row ? p.units * 4 : 0) +
                        ((ngroups + 3) & ~3) * 4 + 32 * 8 + 72 * 4 + p.units + 16;
    cudaError_t e = cudaFuncSetAttribute(alloc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         static_cast<int>(smem));
    if (e != cudaSuccess) return e;
    alloc_kernel<<<p.B, kThreads, smem, stream>>>(p);
    return cudaGetLastError();
}

}  // namespace qs
