/*
 * qstate.h -- C ABI of libqstate: recurrent states of gated linear recurrences stored at low,
 * variable bit width, after "Low-Bit Recurrent States in Hybrid Language Models"
 * (Chen & He, 2026).
 *
 * One head's state S (dk x dv, rows = key channels, columns = value channels) follows Eq. (1):
 *     S_t = (I - k_t a_t^T) D_t S_{t-1} + k_t (w_t o v_t)^T,   o_t = S_t^T q_t,
 *     D_t = diag(e^{-s_t}),
 * with a = beta k, w = beta 1 for KDA and Gated DeltaNet, and a = 0, w = 1 for Mamba-2.
 * Every C tokens (Sec. 2, "Accumulated readout error") the state is written back: quantised
 * with per-unit widths and FP16 range scales (Sec. 3, "Levels and storage") and dequantised
 * before reuse; readouts are taken before quantising.  Widths come from the allocation of
 * Sec. 3 (Eq. 3 weights, Eq. 4 and integer rounding to the layer budget).
 *
 * Conventions for every call:
 *  - Pointers marked "device" are CUDA device pointers owned by the caller; the library never
 *    allocates, frees or retains them.  Host structs are read during the call only.
 *  - `stream` is a cudaStream_t (NULL = legacy default stream).  Work is enqueued
 *    asynchronously on it; the call returns once it is enqueued.
 *  - Arguments are validated on the host before anything is launched.  The return value is
 *    QSTATE_OK or an error code; qstate_last_error() (per host thread) describes the last
 *    failure.  No C++ exception crosses this interface.
 *  - Kernels that find an inconsistent device-side layout (a width above 16, offsets running
 *    past a region, a non-positive decay rate) skip the offending work and set a device status
 *    word; qstate_check() synchronises the stream and reports it.
 *  - All tensors are dense, C-contiguous, float32 unless stated.  Token-major inputs have
 *    shape (B, T, H, d) with T the token extent given in qstate_inputs.
 */
#ifndef QSTATE_H
#define QSTATE_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* ---- status codes ---------------------------------------------------------------------- */
#define QSTATE_OK 0
#define QSTATE_EINVAL 1  /* invalid argument or configuration                                */
#define QSTATE_EBUDGET 2 /* N*bmin > N*bbar or N*bbar > N*bmax: the layer budget is unmeetable */
#define QSTATE_ECUDA 3   /* a CUDA runtime call failed (message in qstate_last_error)          */
#define QSTATE_EDEVICE 4 /* a kernel reported an inconsistent device-side layout or input, or
                            the device was marked unusable (see qstate_check)                 */
#define QSTATE_ETIMEOUT 5 /* a bounded device-side wait gave up (chunked form: a tensor-core
                             product did not signal completion within the wait limit)         */

/* ---- configuration enums ---------------------------------------------------------------- */
#define QSTATE_DECAY_ROW 0   /* one rate per key row (KDA, Sec. 1)                            */
#define QSTATE_DECAY_HEAD 1  /* one rate per head (Gated DeltaNet, Mamba-2)                   */
#define QSTATE_ERASE_DELTA 0 /* a = beta k, w = beta 1 (Eq. 1, KDA / Gated DeltaNet)          */
#define QSTATE_ERASE_NONE 1  /* a = 0, w = 1 (Eq. 1, Mamba-2)                                  */
#define QSTATE_ERASE_GENERAL 2 /* a and w given per token (Eq. 1 in general)                  */
#define QSTATE_UNIT_ROW 0    /* width + FP16 scale per row (Sec. 3, "Allocation units")       */
#define QSTATE_UNIT_HEAD 1   /* width per head, FP16 scale per 32 key rows x value column     */
/* When the allocation of Eq. 3-4 sees its statistics.  LAGGED: the widths a write-back
 * packs with were allocated from the statistics after the previous write-back (qstate_step
 * allocates into `in` after writing `out`).  CURRENT: qstate_step first runs the interval's
 * tokens to get this write-back's ranges and EMAs, allocates from them into out->widths /
 * out->head_off, then packs with those widths (the state and the tokens are processed twice);
 * row unit only. */
#define QSTATE_ALLOC_LAGGED 0
#define QSTATE_ALLOC_CURRENT 1

/* How a write-back interval of C > 1 tokens is computed (same method, same result up to FP32
 * rounding).  TOKEN: token by token (Eq. 1 as written).  CHUNK: in blocks of 16 tokens with
 * the products against the block's starting state and the state update on the tensor cores
 * (3xTF32, FP32 accumulation; Eq. 1 unrolled over the block, Sec. 2's write-back period);
 * row unit, dk = dv = 128, erase_kind DELTA or NONE.  The chunked form needs every row's
 * decay over a 16-token block to stay above FP32's normal range (rates summing to less than
 * about 87 over 16 tokens); a block beyond that sets the device status (QSTATE_EDEVICE from
 * qstate_check).  Calls whose buffers are not 16-byte aligned run the token form. */
#define QSTATE_FORM_TOKEN 0
#define QSTATE_FORM_CHUNK 1

/* Allocation weights c_i (Eq. 3 and the alternatives of Table 1).  With the EMAs of
 * qstate_stats, m_s = EMA(1 - e^{-2s}) and m_r = EMA of the erasure term:
 * Gamma_hat = (1 - m_s) / (expm1(m_r) + m_s); Rtilde^2 = R^2 / mean of R^2 over the unit's
 * output-normalisation group (1 for the head unit, which has no per-unit range, as R is). */
#define QSTATE_WEIGHT_OURS 0      /* Gamma_hat Rtilde^2 (Eq. 3)                                  */
#define QSTATE_WEIGHT_RANGE 1     /* R^2, range alone                                            */
#define QSTATE_WEIGHT_GAMMA_RAW 2 /* Gamma_hat R^2, raw range                                    */
#define QSTATE_WEIGHT_NRANGE 3    /* Rtilde^2, relative range                                    */
#define QSTATE_WEIGHT_PERSIST 4   /* w1 Rtilde^2, persistence w1 = 1/(1 - e^{-2s}) = 1 / m_s      */
#define QSTATE_WEIGHT_WBFACTOR 5  /* h Rtilde^2, write-back factor h = 1/(1 - e^{-2Cs})
                                     = 1 / (1 - (1 - m_s)^C), the power by repeated squaring    */
#define QSTATE_WEIGHT_NOERASE 6   /* Gamma_hat with m_r = 0, times Rtilde^2                      */
#define QSTATE_WEIGHT_SHUFFLE 7   /* Gamma_hat of unit pi(i), times Rtilde_i^2: decay weights
                                     moved to other units by the fixed bijection
                                     pi(i) = (A i + N/3) mod N of the batch element's N units,
                                     A the smallest integer > 0.6180339887 N coprime to N      */
#define QSTATE_WEIGHT_UNIFORM 8   /* equal weights: uniform widths                               */

/* Method configuration.  Sizes: dk in {64, 128}, dv in {64, 128}; dk a multiple of 32 for the
 * head unit; the budget H*dk*dv*bbar must be a whole number of bytes per batch element. */
typedef struct qstate_cfg {
    int32_t B, H, dk, dv;
    int32_t decay_kind;          /* QSTATE_DECAY_*                                           */
    int32_t erase_kind;          /* QSTATE_ERASE_*                                           */
    int32_t unit_kind;           /* QSTATE_UNIT_*; the head unit requires per-head decay     */
    int32_t group_heads;         /* heads per output-normalisation group u(i), row unit (Sec. 2
                                    "Range normalization"); must divide H                    */
    int32_t bbar_num, bbar_den;  /* mean payload bits per element bbar = num/den (Eq. 4)      */
    int32_t bmin, bmax;          /* width limits, 0 <= bmin <= bbar <= bmax <= 16 (Sec. 3)    */
    int32_t C;                   /* write-back period in tokens (Sec. 2), >= 1               */
    int32_t fit_every;           /* 1: fit the range factor f at every write-back (Sec. 3);
                                    K > 1: head h refits when (write-back + h) % K == 0 and
                                    otherwise reuses its stored factor                       */
    float ema_span;              /* EMA span in tokens (Sec. 3: 64)                           */
    int32_t gate_bits;           /* 0: FP32 decay rates; g in 1..8: log-quantised rates       */
    int32_t weight_kind;         /* QSTATE_WEIGHT_*                                          */
    int32_t alloc_mode;          /* QSTATE_ALLOC_LAGGED (0) or QSTATE_ALLOC_CURRENT (1)       */
    int32_t interval_form;       /* QSTATE_FORM_TOKEN (0) or QSTATE_FORM_CHUNK (1)            */
} qstate_cfg;

/* One packed state (device pointers).  Layout (Sec. 3, "Levels and storage"; bit order is
 * this library's reading):
 *  payload  B regions of qstate_region_bytes() bytes.  In region b, head h starts at byte
 *           head_off[b*H + h]; its rows follow in order, row i taking width_i*dv/8 bytes; row
 *           element j's code occupies row bits [j*w, j*w + w), bit m of a row being bit m%8
 *           of byte m/8.  Codes: w >= 2 -> offset binary q + n, n = 2^(w-1) - 1; w = 1 ->
 *           sign bit (1 = negative); w = 0 -> nothing stored.
 *  scales   FP16 bit patterns, one per scale group: (B, H, dk) for the row unit, (B, H, dk/32,
 *           dv) for the head unit.  w >= 2: step Delta; w = 1: mean |x|.
 *  widths   uint8, (B, H, dk) for the row unit, (B, H) for the head unit.
 *  head_off uint32, (B, H), byte offsets inside the batch element's region.
 *  fidx     uint8, one per scale group: index k of the fitted factor f_k = (5 + k)/20. */
typedef struct qstate_buf {
    uint8_t* payload;
    uint16_t* scales;
    uint8_t* widths;
    uint32_t* head_off;
    uint8_t* fidx;
} qstate_buf;

/* Per-unit statistics (device, float32, B*units each; units = H*dk row unit, H head unit):
 *  ema_s  EMA of 1 - e^{-2 s} (the complement of the EMA of the squared decay factor, Sec. 3)
 *  ema_r  EMA of beta (2 - beta) k_i^2 (row unit) or of beta (2 - beta) |k|^2 / dk (head unit)
 *  range  row absolute maximum R_i of the state at the last write-back (row unit only). */
typedef struct qstate_stats {
    float* ema_s;
    float* ema_r;
    float* range;
} qstate_stats;

/* Token inputs (device).  q, k: (B, T, H, dk); v: (B, T, H, dv); s: (B, T, H, dk) for per-row
 * decay or (B, T, H) for per-head decay, all rates > 0; beta: (B, T, H), used by
 * QSTATE_ERASE_DELTA only.  With log-quantised rates pass s = NULL, s_code (uint8, same shape
 * as s) and s_lut (channels x 2^gate_bits levels, channels = H*dk or H) from
 * qstate_quant_decay.  a: (B, T, H, dk) and w: (B, T, H, dv), used by QSTATE_ERASE_GENERAL
 * only: S = (I - k a^T) D S + k (w o v)^T.  Its erasure statistic (the EMA behind Eq. 3's r_i)
 * is 2 a_i k_i - a_i^2 |k|^2, the fraction of row i's error energy one token removes, which
 * is beta (2 - beta) k_i^2 for a = beta k and a unit key (row unit); the head unit averages
 * it over the rows. */
typedef struct qstate_inputs {
    const float* q;
    const float* k;
    const float* v;
    const float* s;
    const uint8_t* s_code;
    const float* s_lut;
    const float* beta;
    int32_t T;
    const float* a;
    const float* w;
} qstate_inputs;

/* ---- sizes and accounting (host only) ---------------------------------------------------- */
/* QSTATE_OK if the configuration is supported; otherwise an error code + message. */
int qstate_validate(const qstate_cfg* cfg);
/* Payload bytes of one batch element: H*dk*dv*bbar/8 (0 if invalid). */
size_t qstate_region_bytes(const qstate_cfg* cfg);
/* Allocation units per batch element (H*dk or H) and scale groups per batch element. */
size_t qstate_units(const qstate_cfg* cfg);
size_t qstate_scale_groups(const qstate_cfg* cfg);
/* Total stored bits per state element (Sec. 3): bbar + (16 + width bits)/dv for the row unit,
 * bbar + 16/32 + width bits/(dk dv) for the head unit; width bits = ceil(log2(bmax-bmin+1)). */
double qstate_bits_per_element(const qstate_cfg* cfg);

/* ---- calls -------------------------------------------------------------------------------- */
/* Initial state (Sec. 3 protocol): widths of the allocation with equal weights (uniform bbar
 * when it is an integer), matching head offsets, and the zero state packed into `a`
 * (scales 0, factor index 15).  `b` receives the same widths and offsets. */
int qstate_init(const qstate_cfg* cfg, qstate_buf* a, qstate_buf* b, void* stream);

/* Sec. 3, Eq. (3) and Eq. (4), followed by the paper's integer step (the real widths are
 * rounded, limited to [b_min, b_max] and corrected until they sum to the layer budget): per
 * batch element, weights c_i = Gamma_hat_i Rtilde_i^2 from `stats`
 * (Gamma_hat = (1 - ema_s)/(expm1(ema_r) + ema_s), Rtilde_i^2 = R_i^2 / mean over the group of
 * R^2, 1 for the head unit) and integer widths summing exactly to units*bbar: the widths that
 * minimise sum_i c_i 4^{-w_i} under the limits, ties going to lower unit indices.  Writes
 * widths_out (B*units) and head_off_out (B*H).  Bit-reproducible. */
int qstate_alloc_bits(const qstate_cfg* cfg, const qstate_stats* stats, uint8_t* widths_out,
                      uint32_t* head_off_out, void* stream);

/* Sec. 3, "Levels and storage": quantise the dense state S (device, (B, H, dk, dv)) with the
 * widths and offsets already in `out` (fitting f for every scale group) and write payload,
 * scales and fidx of `out`; range_out (device, B*units, may be NULL) receives the row absmax. */
int qstate_pack(const qstate_cfg* cfg, const float* S, qstate_buf* out, float* range_out,
                void* stream);

/* Inverse of qstate_pack: dequantise `in` into S_out (device, (B, H, dk, dv)). */
int qstate_unpack(const qstate_cfg* cfg, const qstate_buf* in, float* S_out, void* stream);

/* Sec. 3, "Decay-gate quantization": per channel (h, i) (or per head), levels uniform in
 * log s between the smallest and largest rate over all (b, t): l_k = exp(lo + k (hi-lo)/(L-1)),
 * L = 2^gate_bits, thresholds at the geometric means of neighbours, code = number of
 * thresholds <= s.  s: device (B, T, H, dk) or (B, T, H); code_out: uint8, same shape;
 * lut_out: channels x L levels; thr_out: channels x (L - 1) thresholds.  EDEVICE (from
 * qstate_check) if a rate is not a positive finite number. */
int qstate_quant_decay(const qstate_cfg* cfg, const float* s, int32_t T, uint8_t* code_out,
                       float* lut_out, float* thr_out, void* stream);

/* Same computation and outputs as qstate_quant_decay, for callers that cannot allocate device
 * memory: code running where a device allocation is not allowed or would stall (inside a host
 * framework whose allocator owns all device memory, a plugin that only receives its inputs and
 * outputs, a latency-critical loop that must not call into the allocator).  The paper has no
 * counterpart; it is a deployment convenience.  The thresholds, which qstate_quant_decay writes
 * to thr_out, are kept instead in one fixed array inside the library: at most 65536 thresholds,
 * i.e. channels x (2^gate_bits - 1) <= 65536 (4096 channels at gate_bits = 4); larger
 * configurations return QSTATE_EINVAL with a message and launch nothing.  This call allocates
 * nothing.  The array exists once per device for the life of the process; the first call with a
 * device current looks its address up on the host, so make that first call before any stream
 * capture.  Every call on a device shares the array and leaves its thresholds there; each call
 * rewrites all the entries it reads before reading them, so nothing needs clearing, but calls
 * whose kernels overlap on the GPU (for instance on two streams) race on it. */
int qstate_quant_decay_noalloc(const qstate_cfg* cfg, const float* s, int32_t T,
                               uint8_t* code_out, float* lut_out, void* stream);

/* One write-back interval: tokens [t_begin, t_end) (at most C of them) of every head, from the
 * state packed in `in` to `out` (whose widths and offsets must already hold the target
 * allocation).  Unpack + dequantise, decay, delta update and readout o_t (device,
 * (B, T, H, dv), read before quantising), EMA statistics, range fit, requantise + repack;
 * then the allocation for the next write-back from the new statistics is written into
 * in->widths / in->head_off (in's payload is dead by then), so the next interval runs with
 * the roles of `in` and `out` swapped.  t = 0 initialises the EMAs.  w_index numbers this
 * write-back (for fit_every). */
int qstate_step(const qstate_cfg* cfg, qstate_buf* in, qstate_buf* out,
                const qstate_inputs* x, int32_t t_begin, int32_t t_end, int32_t w_index,
                float* o, qstate_stats* stats, void* stream);

/* Tokens [t_begin, t_end) in write-back intervals of C tokens (the last one may be shorter),
 * ping-ponging between `ping` (holding the state at t_begin, with pong's widths set as the
 * first target) and `pong`.  *final_in_pong is set to 1 if the final state is in `pong`.
 * Equal to the sequence of qstate_step calls, bit for bit.  w_index0 numbers the first
 * write-back. */
int qstate_scan(const qstate_cfg* cfg, qstate_buf* ping, qstate_buf* pong,
                const qstate_inputs* x, int32_t t_begin, int32_t t_end, int32_t w_index0,
                float* o, qstate_stats* stats, int32_t* final_in_pong, void* stream);

/* qstate_scan fed from pinned host memory, for callers whose token inputs and readouts live
 * on the host.  x_host and x_dev describe the same (B, T, H, .) tensors (same T) in host and
 * device memory; every input present in x_host (q, k, v, beta, s or s_code) is copied, token
 * chunk by token chunk, into x_dev's buffer (one copy per tensor, chunk and batch element) on
 * copy_stream, while the compute stream runs the scan of the previous chunk; inputs absent
 * from x_host (e.g. rate codes made on the device by qstate_quant_decay) must already be in
 * x_dev.  Readouts of each chunk are copied from o_dev to o_host once the chunk is done, on a
 * stream the library owns (so that they move while later chunks' inputs come in).  chunk
 * (tokens) is a multiple of C.  stream and copy_stream are distinct non-NULL
 * streams; work on stream completes only after the last readout has reached o_host.  Host
 * memory should be pinned (pageable memory works but the copies then serialise).  Results are
 * those of qstate_scan(ping, pong, x_dev, ...) bit for bit. */
int qstate_scan_host(const qstate_cfg* cfg, qstate_buf* ping, qstate_buf* pong,
                     const qstate_inputs* x_host, const qstate_inputs* x_dev, int32_t t_begin,
                     int32_t t_end, int32_t w_index0, float* o_host, float* o_dev,
                     qstate_stats* stats, int32_t chunk, int32_t* final_in_pong, void* stream,
                     void* copy_stream);

/* Unquantised reference path: Eq. (1) on a dense FP32 state S (device, (B, H, dk, dv), in/out)
 * for tokens [t_begin, t_end), the state round-tripping through memory every C tokens. */
int qstate_scan_fp32(const qstate_cfg* cfg, float* S, const qstate_inputs* x, int32_t t_begin,
                     int32_t t_end, float* o, void* stream);

/* Synchronise `stream`, read and clear the device status word.  QSTATE_OK; QSTATE_ETIMEOUT if a
 * bounded wait of the chunked form gave up (the call's results are not valid; the kernel still
 * waited for its products before freeing tensor memory, so later calls are unaffected);
 * otherwise QSTATE_EDEVICE with the reasons in qstate_last_error().  If even that last wait
 * gave up, tensor memory may have been freed under products in flight: the device is then
 * marked unusable and every later call that launches work on it (and qstate_check) returns
 * QSTATE_EDEVICE for the rest of the process. */
int qstate_check(void* stream);

/* Limit, in polls of the mbarrier, of the chunked form's waits for its tensor-core products in
 * the calls that follow (process-wide; read when a call is enqueued).  polls >= 0 sets it; 0
 * gives up at the first wait without polling (the products still complete, the results of
 * that call are invalid and qstate_check reports QSTATE_ETIMEOUT): a way to exercise the
 * timeout path without a faulty kernel.  polls < 0 restores the default (2^24 polls, far
 * beyond any product's latency).  The wait before freeing tensor memory always uses the
 * default.  Always QSTATE_OK.  Not part of the paper's method: a diagnostic of this library. */
int qstate_set_wait_limit(int32_t polls);

/* Batch partitions of qstate_scan for the calls that follow (process-wide; read when a call is
 * enqueued).  The batch elements of a scan are independent problems (Eq. 1 and the allocation
 * of Sec. 3 act on each element's own state and budget), so a scan may run as n contiguous
 * partitions of the batch, each its own chain of write-back and allocation launches on a
 * library-owned stream, forked from the caller's stream and joined back into it by events
 * before the call's work is complete on that stream; the chains fill each other's idle SMs.
 * The results are bit for bit those of one chain.  n in 1..8 requests n partitions (at most
 * one per batch element, fewer where a partition would start off a 16-byte boundary in any
 * array); 0 (the default) chooses 4 for the token form and 2 for the chunked form.  Calls
 * from several host threads on one device enqueue their partitioned scans one at a time.
 * QSTATE_OK, or QSTATE_EINVAL for n outside 0..8.  Not part of the paper's method: a
 * scheduling choice of this library. */
int qstate_set_scan_partitions(int32_t n);

/* The number of batch partitions qstate_scan would use for these arguments under the current
 * request (1 = one chain on the caller's stream), or 0 if cfg, x or stats is invalid.  No
 * launch. */
int qstate_scan_partition_count(const qstate_cfg* cfg, const qstate_inputs* x, const qstate_stats* stats);

/* Message for the last failure on this host thread ("" if none).  Valid until the next call. */
const char* qstate_last_error(void);

#ifdef __cplusplus
}
#endif
#endif /* QSTATE_H */
