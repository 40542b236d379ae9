// qs_internal.h -- kernel parameter blocks and launch entry points inside libqstate.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include "../../include/qstate.h"

namespace qs {

// device status bits
enum : int {
    QS_DEV_LAYOUT = 1,  // widths/offsets inconsistent with the region
    QS_DEV_RATE = 2,    // a decay rate is not a positive finite number
    QS_DEV_TIMEOUT = 4, // a tensor-core product did not signal completion in time
    QS_DEV_CHUNK = 8,   // chunked form: a row's decay over a 16-token block leaves FP32 range
    QS_DEV_TEARDOWN = 16,  // chunked form: after a timeout, the wait for the products still in
                           // flight before freeing tensor memory also gave up
};

// Default limit of the chunked form's bounded mbarrier waits (polls of mbarrier.try_wait).
constexpr int kDefaultWaitPolls = 1 << 24;

constexpr int kNFit = 16;

// Parameters of the fused write-back kernel.  src/dst are packed or dense depending on the
// kernel instantiation.
struct StepParams {
    int B, H, T;
    int t_begin, t_end, w_index;
    int erase;        // 1: delta rule (a = beta k, w = beta 1); 0: a = 0, w = 1 (or general)
    int general;      // 1: a and w given per token (a_in, w_in)
    int mode;         // 0: full write-back; 1: statistics only (ranges, EMAs, readouts; no
                      // packing); 2: full write-back leaving the EMAs in memory unchanged
    int decay_row;    // 1: per-row rates; 0: per-head rates
    int fit_every;
    int L;            // 2^gate_bits (0 when rates are FP32)
    int group_heads;
    long long region_bytes;
    int stage_bytes;  // shared-memory staging capacity for one head's rows (dk dv bmax / 8)
    float alpha;      // EMA weight 2 / (span + 1)
    int wait_polls;   // limit of the chunked form's waits for its tensor-core products (>= 0)
    // packed source / destination
    const uint8_t* in_payload;
    const uint16_t* in_scales;
    const uint8_t* in_widths;
    const uint32_t* in_head_off;
    const uint8_t* in_fidx;
    uint8_t* out_payload;
    uint16_t* out_scales;
    const uint8_t* out_widths;
    const uint32_t* out_head_off;
    uint8_t* out_fidx;
    // dense source / destination (B, H, dk, dv); src may be null (= zero state)
    const float* dense_in;
    float* dense_out;
    // token inputs
    const float* q;
    const float* k;
    const float* v;
    const float* s;
    const uint8_t* s_code;
    const float* s_lut;
    const float* beta;
    const float* a_in;
    const float* w_in;
    float* o;
    // statistics (may be null when there are no tokens)
    float* ema_s;
    float* ema_r;
    float* range;
    int* status;
};

struct AllocParams {
    int B, H, dk, dv, units, unit_row, group_heads, bmin, bmax;
    long long total;   // sum of widths per batch element
    int uniform;       // 1: ignore statistics, equal weights (initial widths)
    int weight_kind;   // QSTATE_WEIGHT_*
    int C;             // write-back period (write-back factor weight)
    int shuf_a, shuf_b;   // shuffled-decay bijection u -> (shuf_a u + shuf_b) mod units
    const float* ema_s;
    const float* ema_r;
    const float* range;
    uint8_t* widths;
    uint32_t* head_off;
    int* status;
    float e1[17];      // 1/k! (FP64 -> FP32) for the expm1 series, k = 1..16
};

// launchers (return cudaError_t of the launch)
cudaError_t launch_step(const qstate_cfg& cfg, int src_packed, int dst_packed,
                        const StepParams& p, cudaStream_t stream);
cudaError_t launch_alloc(const AllocParams& p, cudaStream_t stream);
cudaError_t launch_quant_decay(const float* s, long long count, int nchan, int g,
                               uint8_t* codes, float* lut, float* thr, int* status,
                               cudaStream_t stream);
long long quant_decay_scratch_capacity();
cudaError_t quant_decay_scratch(float** out);
// identity of the current CUDA context (false if unknown); see qs_api.cu
bool current_context_id(unsigned long long* id);
// streaming multiprocessors of the current device (cached per device)
int device_sm_count();

}  // namespace qs
