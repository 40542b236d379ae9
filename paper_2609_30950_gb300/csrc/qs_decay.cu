// qs_decay.cu -- log-uniform decay-gate quantiser (Sec. 3, "Decay-gate quantization").
//
// Three HBM-bound passes over the rates s (count samples x nchan channels, channel fastest):
//   1. per-channel min / max (integer atomics on the bit patterns: rates are positive floats,
//      whose bit patterns order like the values), accumulated into lut[., 0] and lut[., L-1];
//   2. per channel, FP64 levels l_k = exp(lo + k step) and thresholds
//      exp(lo + (k - 1/2) step), lo/hi = log min/max, step = (hi - lo)/(L - 1), rounded to FP32
//      (l_0 = min and l_{L-1} = max exactly);
//   3. codes = number of thresholds <= s, one byte per rate, 16 rates per thread-iteration.
#include <algorithm>
#include <mutex>

#include "qs_common.cuh"

namespace qs {

namespace {

__global__ void decay_init_kernel(float* lut, int nchan, int L) {
    const int ch = blockIdx.x * blockDim.x + threadIdx.x;
    if (ch < nchan) {
        lut[static_cast<size_t>(ch) * L] = INFINITY;
        lut[static_cast<size_t>(ch) * L + L - 1] = 0.0f;
    }
}

// Thread e0 visits elements e0, e0 + S, e0 + 2S, ... with S a multiple of nchan, so its channel
// is fixed.
__global__ void decay_minmax_kernel(const float* __restrict__ s, long long total, int nchan,
                                    int L, float* lut, int* status) {
    const long long S = static_cast<long long>(gridDim.x) * blockDim.x;
    const long long e0 = static_cast<long long>(blockIdx.x) * blockDim.x + threadIdx.x;
    const int ch = static_cast<int>(e0 % nchan);
    float mn = INFINITY, mx = 0.0f;
    bool bad = false;
    for (long long e = e0; e < total; e += S) {
        const float x = __ldg(s + e);
        if (x > 0.0f && x < INFINITY) {
            mn = fminf(mn, x);
            mx = fmaxf(mx, x);
        } else {
            bad = true;
        }
    }
    if (bad) raise_status(status, QS_DEV_RATE);
    if (e0 < total) {
        atomicMin(reinterpret_cast<int*>(lut + static_cast<size_t>(ch) * L), __float_as_int(mn));
        atomicMax(reinterpret_cast<int*>(lut + static_cast<size_t>(ch) * L + L - 1), __float_as_int(mx));
    }
}

__global__ void decay_levels_kernel(float* lut, float* thr, int nchan, int L, int* status) {
    const int ch = blockIdx.x * blockDim.x + threadIdx.x;
    if (ch >= nchan) return;
    float* l = lut + static_cast<size_t>(ch) * L;
    const float mn = l[0], mx = l[L - 1];
    if (!(mn > 0.0f) || !(mx < INFINITY) || !(mn <= mx)) {
        raise_status(status, QS_DEV_RATE);
        return;
    }
    const double lo = log(static_cast<double>(mn)), hi = log(static_cast<double>(mx));
    const double step = __ddiv_rn(__dsub_rn(hi, lo), static_cast<double>(L - 1));
    for (int k = 1; k < L - 1; ++k) l[k] = static_cast<float>(exp(__dadd_rn(lo, __dmul_rn(static_cast<double>(k), step))));
    for (int k = 1; k < L; ++k)
        thr[static_cast<size_t>(ch) * (L - 1) + k - 1] =
            static_cast<float>(exp(__dadd_rn(lo, __dmul_rn(__dsub_rn(static_cast<double>(k), 0.5), step))));
}

template <int LM1>
__global__ void decay_codes_kernel(const float* __restrict__ s, long long total, int nchan,
                                   const float* __restrict__ thr, uint8_t* __restrict__ codes) {
    // 4 consecutive rates per thread (nchan % 4 == 0 keeps them in one row of channels)
    const long long n4 = total / 4;
    const long long stride = static_cast<long long>(gridDim.x) * blockDim.x;
    for (long long i = static_cast<long long>(blockIdx.x) * blockDim.x + threadIdx.x; i < n4; i += stride) {
        const float4 x = __ldg(reinterpret_cast<const float4*>(s) + i);
        const int ch0 = static_cast<int>((i * 4) % nchan);
        const float xs[4] = {x.x, x.y, x.z, x.w};
        uint32_t packed = 0;
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            const float* t = thr + static_cast<size_t>(ch0 + j) * LM1;
            uint32_t c = 0;
#pragma unroll
            for (int k = 0; k < LM1; ++k) c += (xs[j] >= __ldg(t + k)) ? 1u : 0u;
            packed |= c << (8 * j);
        }
        reinterpret_cast<uint32_t*>(codes)[i] = packed;
    }
}

__global__ void decay_codes_generic_kernel(const float* __restrict__ s, long long total, int nchan,
                                           int LM1, const float* __restrict__ thr,
                                           uint8_t* __restrict__ codes) {
    const long long stride = static_cast<long long>(gridDim.x) * blockDim.x;
    for (long long e = static_cast<long long>(blockIdx.x) * blockDim.x + threadIdx.x; e < total; e += stride) {
        const float x = __ldg(s + e);
        const float* t = thr + static_cast<size_t>(e % nchan) * LM1;
        int c = 0;
        for (int k = 0; k < LM1; ++k) c += (x >= __ldg(t + k)) ? 1 : 0;
        codes[e] = static_cast<uint8_t>(c);
    }
}

long long gcd_ll(long long a, long long b) { return b == 0 ? a : gcd_ll(b, a % b); }

}  // namespace

cudaError_t launch_quant_decay(const float* s, long long count, int nchan, int g, uint8_t* codes,
                               float* lut, float* thr, int* status, cudaStream_t stream) {
    const int L = 1 << g;
    const long long total = count * nchan;
    decay_init_kernel<<<(nchan + 255) / 256, 256, 0, stream>>>(lut, nchan, L);
    // S = a multiple of lcm(nchan, 256) near (SMs x 8) CTAs of 256 threads
    const long long lcm = static_cast<long long>(nchan) / gcd_ll(nchan, 256) * 256;
    const long long target = static_cast<long long>(device_sm_count()) * 8 * 256;
    long long S = std::max(lcm, (target / lcm) * lcm);
    while (S / 256 > 0x7fffffffLL) S -= lcm;
    decay_minmax_kernel<<<static_cast<unsigned>(S / 256), 256, 0, stream>>>(s, total, nchan, L, lut, status);
    decay_levels_kernel<<<(nchan + 127) / 128, 128, 0, stream>>>(lut, thr, nchan, L, status);
    const unsigned blocks = static_cast<unsigned>(device_sm_count()) * 8u;
    if (nchan % 4 == 0 && (reinterpret_cast<uintptr_t>(s) & 15) == 0 &&
        (reinterpret_cast<uintptr_t>(codes) & 3) == 0) {
        switch (L - 1) {
            case 1: decay_codes_kernel<1><<<blocks, 256, 0, stream>>>(s, total, nchan, thr, codes); break;
            case 3: decay_codes_kernel<3><<<blocks, 256, 0, stream>>>(s, total, nchan, thr, codes); break;
            case 7: decay_codes_kernel<7><<<blocks, 256, 0, stream>>>(s, total, nchan, thr, codes); break;
            case 15: decay_codes_kernel<15><<<blocks, 256, 0, stream>>>(s, total, nchan, thr, codes); break;
            default:
                decay_codes_generic_kernel<<<blocks, 256, 0, stream>>>(s, total, nchan, L - 1, thr, codes);
        }
    } else {
        decay_codes_generic_kernel<<<blocks, 256, 0, stream>>>(s, total, nchan, L - 1, thr, codes);
    }
    return cudaGetLastError();
}

// ---- variant without caller-supplied threshold buffer -------------------------------------------
// The thresholds are an intermediate of the quantiser.  Callers that must not allocate device
// memory of their own keep them here: one file-scope array per device (every GPU that loads
// the library holds it until the process exits), shared by all calls on that device.
constexpr long long kDecayScratchFloats = 65536;   // 256 KiB: channels x (2^g - 1) thresholds
static __device__ __align__(256) float g_decay_thr_scratch[kDecayScratchFloats];

namespace {
constexpr int kMaxDev = 64;
std::mutex g_scratch_mu;
float* g_scratch_addr[kMaxDev] = {};
unsigned long long g_scratch_ctx[kMaxDev] = {};
}  // namespace

long long quant_decay_scratch_capacity() { return kDecayScratchFloats; }

// Device address of the threshold scratch on the current device, looked up on the first call
// made with that device current (a host-side lookup: make it before any stream capture), and
// again whenever the device's context has been created anew since (its module, and with it
// the array, may then sit at another address).
cudaError_t quant_decay_scratch(float** out) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= kMaxDev) return cudaErrorInvalidDevice;
    std::lock_guard<std::mutex> lock(g_scratch_mu);
    unsigned long long ctx = 0;
    const bool known = current_context_id(&ctx);
    if (!g_scratch_addr[dev] || !known || ctx != g_scratch_ctx[dev]) {
        void* ptr = nullptr;
        e = cudaGetSymbolAddress(&ptr, g_decay_thr_scratch);
        if (e != cudaSuccess) return e;
        g_scratch_addr[dev] = static_cast<float*>(ptr);
        g_scratch_ctx[dev] = current_context_id(&ctx) ? ctx : 0ull;
    }
    *out = g_scratch_addr[dev];
    return cudaSuccess;
}

}  // namespace qs
