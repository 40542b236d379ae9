// qs_common.cuh -- device helpers shared by the libqstate kernels (sm_103a).
//
// Floating-point operations that decide an integer (a code, a fitted factor, a width) are
// written with explicit IEEE intrinsics (__fmul_rn, __fadd_rn, __frcp_rn, ...) so that the
// compiler cannot contract them into FMAs: the stored format is then reproducible.
#pragma once

#include <cuda_fp16.h>
#include <stdint.h>

#include "qs_internal.h"

namespace qs {

constexpr unsigned kFull = 0xffffffffu;
// 1.5 * 2^23: y + kMagic rounds y to an integer (round-half-even) for |y| < 2^22, and the
// result's low mantissa bits hold that integer offset by 2^22.
constexpr float kMagic = 12582912.0f;
constexpr uint32_t kMagicBits = 0x4B400000u;
// 2^23: the float with bits 0x4B000000 | u equals 2^23 + u for u < 2^23.
constexpr uint32_t kTwo23Bits = 0x4B000000u;

// Record a QS_DEV_* condition in the status word (one per device, see qs_api.cu).
__device__ __forceinline__ void raise_status(int* status, int bits) {
    if (status) atomicOr(status, bits);
}

// ---- FP16 scale (Sec. 3, "Levels and storage") -------------------------------------------
// Round to binary16 (nearest even), magnitudes saturated at 65504, returned as float.
__device__ __forceinline__ float f16_round(float x) {
    x = fminf(fmaxf(x, -65504.0f), 65504.0f);
    return __half2float(__float2half_rn(x));
}
__device__ __forceinline__ uint16_t f16_bits(float x) {
    x = fminf(fmaxf(x, -65504.0f), 65504.0f);
    return __half_as_ushort(__float2half_rn(x));
}
__device__ __forceinline__ float f16_value(uint16_t u) { return __half2float(__ushort_as_half(u)); }

// The 16 candidate range factors f_k = (5 + k) / 20 on [1/4, 1] (Sec. 3), correctly rounded.
__device__ __forceinline__ float fit_factor(int k) {
    return __fdiv_rn(static_cast<float>(5 + k), 20.0f);
}

// Candidate step for factor f: Delta = FP16(fl(fl(f R) * fl(1/n))).
__device__ __forceinline__ float cand_step(float f, float R, float inv_n) {
    return f16_round(__fmul_rn(__fmul_rn(f, R), inv_n));
}
__device__ __forceinline__ float step_rcp(float D) { return D == 0.0f ? 0.0f : __frcp_rn(D); }

// clamp(rint(x * inv), -n, n) in the magic domain: returns kMagic + q (exact integer float).
__device__ __forceinline__ float code_magic(float x, float inv, float lo, float hi) {
    float t = __fadd_rn(__fmul_rn(x, inv), kMagic);
    return fminf(fmaxf(t, lo), hi);
}

// Erasure statistic of a row under general erasure (Eq. (1) with a given a):
// 2 a_i k_i - a_i^2 |k|^2, the fraction of the row's error energy that (I - k a^T) removes;
// |k|^2 summed in index order over the DK entries of kvec, one rounding per operation.
template <int DK>
__device__ __forceinline__ float general_erasure(float ai, float ki, const float* kvec) {
    float ksq = 0.0f;
#pragma unroll 8
    for (int r = 0; r < DK; ++r) ksq = __fadd_rn(ksq, __fmul_rn(kvec[r], kvec[r]));
    return __fsub_rn(__fmul_rn(2.0f, __fmul_rn(ai, ki)), __fmul_rn(__fmul_rn(ai, ai), ksq));
}

// ---- warp reductions ----------------------------------------------------------------------
__device__ __forceinline__ float warp_absmax(float v) {
    unsigned m = __reduce_max_sync(kFull, __float_as_uint(fabsf(v)));
    return __uint_as_float(m);
}
__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(kFull, v, o);
    return v;
}

// ---- row bitstream (Sec. 3 storage; this library's bit order) ------------------------------
// A lane owning CPL consecutive elements of a row reads its CPL*w bits starting at row bit
// lane*CPL*w.  `row` is 8-byte aligned shared memory followed by >= 12 readable bytes.
template <int CPL>
__device__ __forceinline__ void extract_codes(const uint8_t* row, int lane, int w,
                                              uint32_t (&u)[CPL]) {
    const uint32_t* words = reinterpret_cast<const uint32_t*>(row);
    const int P = lane * CPL * w;
    const int idx = P >> 5, sh = P & 31;
    const uint32_t mask = (w >= 32) ? 0xffffffffu : ((1u << w) - 1u);
    if (CPL * w <= 32) {
        uint32_t chunk = __funnelshift_r(words[idx], words[idx + 1], sh);
#pragma unroll
        for (int c = 0; c < CPL; ++c) u[c] = (chunk >> (c * w)) & mask;
    } else {
        uint32_t lo = __funnelshift_r(words[idx], words[idx + 1], sh);
        uint32_t hi = __funnelshift_r(words[idx + 1], words[idx + 2], sh);
        uint64_t chunk = (static_cast<uint64_t>(hi) << 32) | lo;
#pragma unroll
        for (int c = 0; c < CPL; ++c) u[c] = static_cast<uint32_t>(chunk >> (c * w)) & mask;
    }
}

}  // namespace qs
