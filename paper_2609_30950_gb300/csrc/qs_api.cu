// qs_api.cu -- the C ABI of libqstate (declared in include/qstate.h): host-side validation,
// error reporting and kernel dispatch.
#include <cuda.h>   // driver types only (CUcontext); entry points come through the runtime

#include <atomic>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <mutex>

#include "qs_internal.h"

namespace qs {
cudaError_t launch_step_128x128(const qstate_cfg&, int, int, const StepParams&, cudaStream_t);
cudaError_t launch_step_128x64(const qstate_cfg&, int, int, const StepParams&, cudaStream_t);
cudaError_t launch_step_64x64(const qstate_cfg&, int, int, const StepParams&, cudaStream_t);
cudaError_t launch_wb_row_128x128(const qstate_cfg&, const StepParams&, cudaStream_t);
cudaError_t launch_wb_row_128x64(const qstate_cfg&, const StepParams&, cudaStream_t);
cudaError_t launch_wb_row_64x64(const qstate_cfg&, const StepParams&, cudaStream_t);
cudaError_t launch_wb_chunk_128x128(const qstate_cfg&, const StepParams&, cudaStream_t);

// Streaming multiprocessors of the current device, queried once per device.
int device_sm_count() {
    static std::atomic<int> cache[64] = {};
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 1;
    int n = cache[dev].load();
    if (n <= 0) {
        if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0) return 1;
        cache[dev].store(n);
    }
    return n;
}

// Identity of the calling thread's current CUDA context (cuCtxGetId), fetched through the
// runtime so that the library does not link the driver library.  A context that is destroyed
// and created again (cudaDeviceReset, a primary-context reset by a host framework) gets a new
// identity, and with it the module holding this library's device variables may be loaded at
// new addresses: host-side caches of those addresses are keyed on it.  False if there is no
// current context or the driver lacks the call.
bool current_context_id(unsigned long long* id) {
    using GetCurrent = CUresult (*)(CUcontext*);
    using GetId = CUresult (*)(CUcontext, unsigned long long*);
    static GetCurrent get_current = nullptr;
    static GetId get_id = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        void* f = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &f, 12000, cudaEnableDefault, &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            get_current = reinterpret_cast<GetCurrent>(f);
        f = nullptr;
        if (cudaGetDriverEntryPointByVersion("cuCtxGetId", &f, 12000, cudaEnableDefault, &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            get_id = reinterpret_cast<GetId>(f);
    });
    if (!get_current || !get_id) return false;
    CUcontext ctx = nullptr;
    if (get_current(&ctx) != CUDA_SUCCESS || ctx == nullptr) return false;
    return get_id(ctx, id) == CUDA_SUCCESS;
}

}  // namespace qs

using namespace qs;

// Device status word (QS_DEV_* bits).  Kernels receive its address; see status_word().
static __device__ int qs_status_word;

namespace {

thread_local char g_err[512] = "";

int fail(int code, const char* fmt, ...) {
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(g_err, sizeof(g_err), fmt, ap);
    va_end(ap);
    return code;
}

int cuda_fail(cudaError_t e, const char* what) {
    return fail(QSTATE_ECUDA, "%s: %s (%s)", what, cudaGetErrorName(e), cudaGetErrorString(e));
}

constexpr int kMaxDevices = 64;
std::mutex g_mu;
// per device: the status word's address and the context it was looked up in
int* g_status_addr[kMaxDevices] = {};
unsigned long long g_status_ctx[kMaxDevices] = {};
// Devices on which a chunked-form teardown wait gave up (QS_DEV_TEARDOWN): tensor memory may
// have been freed under products still in flight, so later results could not be trusted and
// every launching call is refused for the rest of the process.
std::atomic<bool> g_unusable[kMaxDevices] = {};
// Limit of the chunked form's mbarrier waits for the following launches (qstate_set_wait_limit).
std::atomic<int> g_wait_polls{kDefaultWaitPolls};

// Address of the status word on the current device, looked up once per device and context
// (again whenever the context's identity is unknown or has changed).
int* status_word(cudaError_t* err, int* dev_out = nullptr) {
    int dev = 0;
    *err = cudaGetDevice(&dev);
    if (*err != cudaSuccess || dev < 0 || dev >= kMaxDevices) return nullptr;
    if (dev_out) *dev_out = dev;
    std::lock_guard<std::mutex> lock(g_mu);
    unsigned long long ctx = 0;
    const bool known = current_context_id(&ctx);
    if (!g_status_addr[dev] || !known || ctx != g_status_ctx[dev]) {
        void* p = nullptr;
        *err = cudaGetSymbolAddress(&p, qs_status_word);
        if (*err != cudaSuccess) return nullptr;
        g_status_addr[dev] = static_cast<int*>(p);
        // the lookup makes the context current if it was not yet
        g_status_ctx[dev] = current_context_id(&ctx) ? ctx : 0ull;
    }
    return g_status_addr[dev];
}

// The status word of the current device for a call that launches work; refused (EDEVICE) once
// the device has been marked unusable.
int acquire_status(int** out) {
    cudaError_t e = cudaSuccess;
    int dev = -1;
    int* p = status_word(&e, &dev);
    if (!p) return cuda_fail(e, "status word");
    if (g_unusable[dev].load())
        return fail(QSTATE_EDEVICE, "device %d is marked unusable: a tensor-core teardown wait gave up "
                    "earlier in this process", dev);
    *out = p;
    return QSTATE_OK;
}

long long units_of(const qstate_cfg* c) {
    return c->unit_kind == QSTATE_UNIT_ROW ? static_cast<long long>(c->H) * c->dk : c->H;
}
long long groups_of(const qstate_cfg* c) {
    return c->unit_kind == QSTATE_UNIT_ROW ? static_cast<long long>(c->H) * c->dk
                                           : static_cast<long long>(c->H) * (c->dk / 32) * c->dv;
}

int validate(const qstate_cfg* c) {
    if (!c) return fail(QSTATE_EINVAL, "cfg is NULL");
    if (c->B < 1 || c->H < 1 || c->H > 1024) return fail(QSTATE_EINVAL, "need B >= 1 and 1 <= H <= 1024");
    const bool shape_ok = (c->dk == 128 && c->dv == 128) || (c->dk == 128 && c->dv == 64) ||
                          (c->dk == 64 && c->dv == 64);
    if (!shape_ok) return fail(QSTATE_EINVAL, "unsupported (dk, dv) = (%d, %d)", c->dk, c->dv);
    if (c->decay_kind != QSTATE_DECAY_ROW && c->decay_kind != QSTATE_DECAY_HEAD)
        return fail(QSTATE_EINVAL, "bad decay_kind");
    if (c->erase_kind != QSTATE_ERASE_DELTA && c->erase_kind != QSTATE_ERASE_NONE &&
        c->erase_kind != QSTATE_ERASE_GENERAL)
        return fail(QSTATE_EINVAL, "bad erase_kind");
    if (c->unit_kind != QSTATE_UNIT_ROW && c->unit_kind != QSTATE_UNIT_HEAD)
        return fail(QSTATE_EINVAL, "bad unit_kind");
    if (c->unit_kind == QSTATE_UNIT_HEAD && c->decay_kind != QSTATE_DECAY_HEAD)
        return fail(QSTATE_EINVAL, "the head unit needs per-head decay");
    if (c->unit_kind == QSTATE_UNIT_ROW && (c->group_heads < 1 || c->H % c->group_heads != 0))
        return fail(QSTATE_EINVAL, "group_heads must divide H");
    if (c->bbar_den < 1 || c->bbar_num < 0) return fail(QSTATE_EINVAL, "bad bbar fraction");
    if (c->bmin < 0 || c->bmax > 16 || c->bmin > c->bmax) return fail(QSTATE_EINVAL, "need 0 <= bmin <= bmax <= 16");
    const long long bits = static_cast<long long>(c->H) * c->dk * c->dv * c->bbar_num;
    if (bits % (8LL * c->bbar_den) != 0) return fail(QSTATE_EINVAL, "budget is not a whole number of bytes");
    const long long N = units_of(c);
    if ((N * c->bbar_num) % c->bbar_den != 0) return fail(QSTATE_EINVAL, "units * bbar is not an integer");
    const long long total = N * c->bbar_num / c->bbar_den;
    if (N * c->bmin > total || N * c->bmax < total)
        return fail(QSTATE_EBUDGET, "budget %lld bits per element sum outside [%lld, %lld]", total,
                    N * c->bmin, N * c->bmax);
    if (N > 16384) return fail(QSTATE_EINVAL, "at most 16384 allocation units per batch element");
    if (c->C < 1) return fail(QSTATE_EINVAL, "C must be >= 1");
    if (c->fit_every < 1) return fail(QSTATE_EINVAL, "fit_every must be >= 1");
    if (!(c->ema_span > 0.0f)) return fail(QSTATE_EINVAL, "ema_span must be > 0");
    if (c->gate_bits < 0 || c->gate_bits > 8) return fail(QSTATE_EINVAL, "gate_bits must be in [0, 8]");
    if (c->alloc_mode != QSTATE_ALLOC_LAGGED && c->alloc_mode != QSTATE_ALLOC_CURRENT)
        return fail(QSTATE_EINVAL, "unsupported alloc_mode %d", c->alloc_mode);
    if (c->alloc_mode == QSTATE_ALLOC_CURRENT && c->unit_kind != QSTATE_UNIT_ROW)
        return fail(QSTATE_EINVAL, "alloc_mode current is for the row unit");
    if (c->weight_kind < QSTATE_WEIGHT_OURS || c->weight_kind > QSTATE_WEIGHT_UNIFORM)
        return fail(QSTATE_EINVAL, "unsupported weight_kind %d", c->weight_kind);
    if (c->interval_form != QSTATE_FORM_TOKEN && c->interval_form != QSTATE_FORM_CHUNK)
        return fail(QSTATE_EINVAL, "unsupported interval_form %d", c->interval_form);
    if (c->interval_form == QSTATE_FORM_CHUNK &&
        (c->unit_kind != QSTATE_UNIT_ROW || c->dk != 128 || c->dv != 128 || c->erase_kind == QSTATE_ERASE_GENERAL))
        return fail(QSTATE_EINVAL, "the chunked form needs the row unit, dk = dv = 128 and erase DELTA or NONE");
    return QSTATE_OK;
}

long long region_of(const qstate_cfg* c) {
    return static_cast<long long>(c->H) * c->dk * c->dv * c->bbar_num / (8LL * c->bbar_den);
}

bool buf_ok(const qstate_buf* b) {
    return b && b->payload && b->scales && b->widths && b->head_off && b->fidx;
}

cudaError_t launch_step_any(const qstate_cfg& c, int src_packed, int dst_packed, const StepParams& p,
                            cudaStream_t st) {
    if (c.dk == 128 && c.dv == 128) return launch_step_128x128(c, src_packed, dst_packed, p, st);
    if (c.dk == 128 && c.dv == 64) return launch_step_128x64(c, src_packed, dst_packed, p, st);
    return launch_step_64x64(c, src_packed, dst_packed, p, st);
}

bool aligned16(const void* ptr) { return (reinterpret_cast<uintptr_t>(ptr) & 15u) == 0; }

// The persistent row-unit write-back kernel copies its inputs with 16-byte cp.async and needs
// every per-head array 16-byte aligned; otherwise the one-head-per-CTA kernel runs.
bool wb_row_eligible(const qstate_cfg& c, const StepParams& p) {
    if (c.unit_kind != QSTATE_UNIT_ROW) return false;
    const void* ptrs[] = {p.in_payload, p.in_scales, p.in_widths, p.in_fidx, p.out_payload,
                          p.out_widths, p.q, p.k, p.v, p.ema_s, p.ema_r,
                          p.s_code ? static_cast<const void*>(p.s_code) : static_cast<const void*>(p.s)};
    for (const void* q : ptrs)
        if (q && !aligned16(q)) return false;
    if (!p.in_fidx) return false;
    if (p.decay_row && p.s_code == nullptr && p.s == nullptr) return false;
    return true;
}

cudaError_t launch_writeback(const qstate_cfg& c, const StepParams& p, cudaStream_t st) {
    if (wb_row_eligible(c, p)) {
        if (c.interval_form == QSTATE_FORM_CHUNK && c.dk == 128 && c.dv == 128 && !p.general)
            return launch_wb_chunk_128x128(c, p, st);
        if (c.dk == 128 && c.dv == 128) return launch_wb_row_128x128(c, p, st);
        if (c.dk == 128 && c.dv == 64) return launch_wb_row_128x64(c, p, st);
        return launch_wb_row_64x64(c, p, st);
    }
    return launch_step_any(c, 1, 1, p, st);
}

StepParams base_params(const qstate_cfg* c, int* status) {
    StepParams p;
    std::memset(&p, 0, sizeof(p));
    p.B = c->B;
    p.H = c->H;
    p.erase = c->erase_kind == QSTATE_ERASE_DELTA ? 1 : 0;
    p.general = c->erase_kind == QSTATE_ERASE_GENERAL ? 1 : 0;
    p.decay_row = c->decay_kind == QSTATE_DECAY_ROW ? 1 : 0;
    p.fit_every = c->fit_every;
    p.L = c->gate_bits > 0 ? (1 << c->gate_bits) : 0;
    p.group_heads = c->group_heads;
    p.region_bytes = region_of(c);
    p.alpha = 2.0f / (c->ema_span + 1.0f);
    p.wait_polls = g_wait_polls.load();
    p.status = status;
    return p;
}

int check_inputs(const qstate_cfg* c, const qstate_inputs* x, int t_begin, int t_end, const float* o) {
    if (!x || !x->q || !x->k || !x->v || !o) return fail(QSTATE_EINVAL, "null input or output pointer");
    if (c->erase_kind == QSTATE_ERASE_DELTA && !x->beta) return fail(QSTATE_EINVAL, "beta is NULL");
    if (c->erase_kind == QSTATE_ERASE_GENERAL && (!x->a || !x->w))
        return fail(QSTATE_EINVAL, "general erasure needs a and w");
    if (x->s_code) {
        if (c->gate_bits < 1 || !x->s_lut) return fail(QSTATE_EINVAL, "s_code needs gate_bits >= 1 and s_lut");
    } else if (!x->s) {
        return fail(QSTATE_EINVAL, "decay rates are NULL");
    }
    if (t_begin < 0 || t_end < t_begin || t_end > x->T) return fail(QSTATE_EINVAL, "bad token range");
    return QSTATE_OK;
}

void set_inputs(StepParams& p, const qstate_inputs* x) {
    p.T = x->T;
    p.q = x->q;
    p.k = x->k;
    p.v = x->v;
    p.s = x->s_code ? nullptr : x->s;
    p.s_code = x->s_code;
    p.s_lut = x->s_lut;
    p.beta = x->beta;
    p.a_in = x->a;
    p.w_in = x->w;
}

// Staging of token chunks between pinned host memory and the device: tokens [t0, t1) of every
// batch element of a (B, T, per-token bytes) tensor, 16 bytes per thread and step.  The host
// side is read or written in place (pinned memory is mapped into the device address space), so
// one small launch replaces B row copies; it needs few registers and no shared memory and so
// shares SMs with the write-back kernel.
__global__ void __launch_bounds__(128) stage_tokens_kernel(uint4* dst, const uint4* src, int B,
                                                           long long pitch16, long long off16,
                                                           long long width16) {
    const long long n = static_cast<long long>(B) * width16;
    for (long long e = static_cast<long long>(blockIdx.x) * blockDim.x + threadIdx.x; e < n;
         e += static_cast<long long>(gridDim.x) * blockDim.x) {
        const long long b = e / width16, c = e - b * width16;
        dst[b * pitch16 + off16 + c] = src[b * pitch16 + off16 + c];
    }
}

// The shuffled-decay bijection of N units: u -> (A u + N / 3) mod N with A the smallest
// integer above 0.6180339887 N that is coprime to N.
int gcd_int(int a, int b) { return b == 0 ? a : gcd_int(b, a % b); }
void shuffle_params(int N, int* A, int* Bo) {
    int a = static_cast<int>(0.6180339887 * N) + 1;
    while (gcd_int(a, N) != 1) ++a;
    *A = a % N;
    *Bo = N / 3;
}

int run_alloc(const qstate_cfg* c, const float* ms, const float* mr, const float* range, int uniform,
              uint8_t* widths, uint32_t* head_off, int* status, cudaStream_t st) {
    AllocParams a;
    std::memset(&a, 0, sizeof(a));
    a.B = c->B;
    a.H = c->H;
    a.dk = c->dk;
    a.dv = c->dv;
    a.units = static_cast<int>(units_of(c));
    a.unit_row = c->unit_kind == QSTATE_UNIT_ROW ? 1 : 0;
    a.group_heads = c->unit_kind == QSTATE_UNIT_ROW ? c->group_heads : 1;
    a.bmin = c->bmin;
    a.bmax = c->bmax;
    a.total = units_of(c) * c->bbar_num / c->bbar_den;
    a.uniform = uniform || c->weight_kind == QSTATE_WEIGHT_UNIFORM;
    a.weight_kind = c->weight_kind;
    a.C = c->C;
    shuffle_params(a.units, &a.shuf_a, &a.shuf_b);
    a.ema_s = ms;
    a.ema_r = mr;
    a.range = range;
    a.widths = widths;
    a.head_off = head_off;
    a.status = status;
    double fact = 1.0;
    for (int k = 1; k <= 16; ++k) {
        fact *= static_cast<double>(k);
        a.e1[k] = static_cast<float>(1.0 / fact);
    }
    cudaError_t e = launch_alloc(a, st);
    return e == cudaSuccess ? QSTATE_OK : cuda_fail(e, "allocation kernel");
}

// ---- a scan as concurrent batch partitions ------------------------------------------------------
// The batch elements of a scan are independent problems: Eq. (1), the statistics and the
// allocation of Sec. 3 act on each element's own state and budget.  qstate_scan may therefore
// run G contiguous batch partitions, each a chain of write-back and allocation launches on a
// stream of its own, forked from the caller's stream and joined back into it by events.  The
// chains fill each other's idle SMs (the last wave of a launch, and the allocation launches,
// which occupy one CTA per batch element).  Every kernel computes each head and batch element on
// its own, so the results are those of one chain bit for bit.
constexpr int kMaxParts = 8;
struct PartStreams {
    bool ready = false;
    unsigned long long ctx = 0;
    cudaStream_t s[kMaxParts] = {};          // s[0] unused: partition 0 runs on the caller's stream
    cudaStream_t rd = nullptr;               // qstate_scan_host's readout copies
    cudaEvent_t fork = nullptr;
    cudaEvent_t join[kMaxParts] = {};
};
PartStreams g_parts[kMaxDevices];
// The fork and join events are shared by the calls on a device: a partitioned scan is enqueued
// under this lock (the enqueue only, not the work).
std::mutex g_part_mu;
// Partitions requested by qstate_set_scan_partitions (0: chosen per configuration).
std::atomic<int> g_scan_parts{0};

// Streams and events of the current device, created once per device and context.  Caller holds
// g_part_mu.
int part_streams(PartStreams** out) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return cuda_fail(e, "cudaGetDevice");
    if (dev < 0 || dev >= kMaxDevices) return fail(QSTATE_EDEVICE, "device index %d out of range", dev);
    unsigned long long ctx = 0;
    const bool known = current_context_id(&ctx);
    PartStreams& P = g_parts[dev];
    if (!P.ready || !known || ctx != P.ctx) {
        // handles of an earlier context went with it; nothing to destroy
        P = PartStreams{};
        for (int i = 1; i < kMaxParts; ++i)
            if ((e = cudaStreamCreateWithFlags(&P.s[i], cudaStreamNonBlocking)) != cudaSuccess)
                return cuda_fail(e, "partition stream");
        if ((e = cudaStreamCreateWithFlags(&P.rd, cudaStreamNonBlocking)) != cudaSuccess)
            return cuda_fail(e, "readout stream");
        if ((e = cudaEventCreateWithFlags(&P.fork, cudaEventDisableTiming)) != cudaSuccess)
            return cuda_fail(e, "partition event");
        for (int i = 1; i < kMaxParts; ++i)
            if ((e = cudaEventCreateWithFlags(&P.join[i], cudaEventDisableTiming)) != cudaSuccess)
                return cuda_fail(e, "partition event");
        P.ctx = known ? ctx : 0ull;
        P.ready = known;   // an unknown context is asked again next time
    }
    *out = &P;
    return QSTATE_OK;
}

// Bytes per batch element of every array a scan touches, with the partition's view of them.
struct ScanArrays {
    qstate_buf ping, pong;
    qstate_inputs x;
    float* o;
    qstate_stats st;
};

long long elem_offset_low_bits(const qstate_cfg* c, const qstate_inputs* x, const qstate_stats* st,
                                      long long b0) {
    // OR of the byte offsets of batch element b0 in every array: 16-byte aligned iff its low
    // four bits are zero
    const long long T = x->T, H = c->H, dk = c->dk, dv = c->dv;
    const long long units = units_of(c), groups = groups_of(c);
    const long long ns = c->decay_kind == QSTATE_DECAY_ROW ? T * H * dk : T * H;
    long long m = b0 * region_of(c);
    m |= b0 * groups * 2;
    m |= b0 * units;
    m |= b0 * H * 4;
    m |= b0 * groups;
    if (st) m |= b0 * units * 4;
    m |= b0 * T * H * dk * 4;
    m |= b0 * T * H * dv * 4;
    m |= x->s_code ? b0 * ns : b0 * ns * 4;
    if (x->beta) m |= b0 * T * H * 4;
    return m & 15;
}

ScanArrays slice(const qstate_cfg* c, const qstate_buf* ping, const qstate_buf* pong, const qstate_inputs* x,
                 float* o, const qstate_stats* st, long long b0) {
    const long long T = x->T, H = c->H, dk = c->dk, dv = c->dv;
    const long long units = units_of(c), groups = groups_of(c), region = region_of(c);
    const long long ns = c->decay_kind == QSTATE_DECAY_ROW ? T * H * dk : T * H;
    auto buf = [&](const qstate_buf* b) {
        qstate_buf r;
        r.payload = b->payload + b0 * region;
        r.scales = b->scales + b0 * groups;
        r.widths = b->widths + b0 * units;
        r.head_off = b->head_off + b0 * H;
        r.fidx = b->fidx + b0 * groups;
        return r;
    };
    ScanArrays a;
    a.ping = buf(ping);
    a.pong = buf(pong);
    a.x = *x;
    a.x.q = x->q + b0 * T * H * dk;
    a.x.k = x->k + b0 * T * H * dk;
    a.x.v = x->v + b0 * T * H * dv;
    if (x->s) a.x.s = x->s + b0 * ns;
    if (x->s_code) a.x.s_code = x->s_code + b0 * ns;
    if (x->beta) a.x.beta = x->beta + b0 * T * H;
    if (x->a) a.x.a = x->a + b0 * T * H * dk;
    if (x->w) a.x.w = x->w + b0 * T * H * dv;
    a.o = o + b0 * T * H * dv;
    a.st.ema_s = st->ema_s + b0 * units;
    a.st.ema_r = st->ema_r + b0 * units;
    a.st.range = st->range ? st->range + b0 * units : nullptr;
    return a;
}

// Partitions of a scan: the requested number, else the count measured best on GB300 for the
// benchmark layer shapes (token form 4: 6 % per token at KDA decode, 24 % at Gated DeltaNet;
// chunked form 2: 10 % at KDA prefill, where 3 or 4 split its 16 batch elements less evenly over
// the one-CTA-per-SM launches); at most one per batch element, and fewer where a partition would
// start off a 16-byte boundary in any array.
int scan_parts(const qstate_cfg* c, const qstate_inputs* x, const qstate_stats* st) {
    int G = g_scan_parts.load();
    if (G <= 0) G = c->interval_form == QSTATE_FORM_CHUNK ? 2 : 4;
    G = G < kMaxParts ? G : kMaxParts;
    G = G < c->B ? G : c->B;
    for (; G > 1; --G) {
        bool ok = true;
        for (int p = 1; p < G && ok; ++p)
            ok = elem_offset_low_bits(c, x, st, static_cast<long long>(c->B) * p / G) == 0;
        if (ok) break;
    }
    return G;
}

}  // namespace

extern "C" {

int qstate_validate(const qstate_cfg* cfg) { return validate(cfg); }

size_t qstate_region_bytes(const qstate_cfg* cfg) {
    return validate(cfg) == QSTATE_OK ? static_cast<size_t>(region_of(cfg)) : 0;
}

size_t qstate_units(const qstate_cfg* cfg) {
    return validate(cfg) == QSTATE_OK ? static_cast<size_t>(units_of(cfg)) : 0;
}

size_t qstate_scale_groups(const qstate_cfg* cfg) {
    return validate(cfg) == QSTATE_OK ? static_cast<size_t>(groups_of(cfg)) : 0;
}

double qstate_bits_per_element(const qstate_cfg* cfg) {
    if (validate(cfg) != QSTATE_OK) return 0.0;
    const double bbar = static_cast<double>(cfg->bbar_num) / cfg->bbar_den;
    int wbits = 0;
    while ((1 << wbits) < cfg->bmax - cfg->bmin + 1) ++wbits;
    if (cfg->unit_kind == QSTATE_UNIT_ROW) return bbar + (16.0 + wbits) / cfg->dv;
    return bbar + 0.5 + static_cast<double>(wbits) / (static_cast<double>(cfg->dk) * cfg->dv);
}

int qstate_init(const qstate_cfg* cfg, qstate_buf* a, qstate_buf* b, void* stream) {
    int rc = validate(cfg);
    if (rc) return rc;
    if (!buf_ok(a) || !buf_ok(b)) return fail(QSTATE_EINVAL, "null buffer pointer");
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    int* status = nullptr;
    if ((rc = acquire_status(&status))) return rc;
    cudaError_t e;
    rc = run_alloc(cfg, nullptr, nullptr, nullptr, 1, a->widths, a->head_off, status, st);
    if (rc) return rc;
    const size_t nw = static_cast<size_t>(cfg->B) * units_of(cfg);
    e = cudaMemcpyAsync(b->widths, a->widths, nw, cudaMemcpyDeviceToDevice, st);
    if (e == cudaSuccess)
        e = cudaMemcpyAsync(b->head_off, a->head_off, sizeof(uint32_t) * cfg->B * cfg->H,
                            cudaMemcpyDeviceToDevice, st);
    if (e != cudaSuccess) return cuda_fail(e, "copy of initial widths");
    StepParams p = base_params(cfg, status);
    p.fit_every = 1;
    p.out_payload = a->payload;
    p.out_scales = a->scales;
    p.out_widths = a->widths;
    p.out_head_off = a->head_off;
    p.out_fidx = a->fidx;
    e = launch_step_any(*cfg, 0, 1, p, st);   // dense zero state -> packed
    return e == cudaSuccess ? QSTATE_OK : cuda_fail(e, "pack kernel");
}

int qstate_alloc_bits(const qstate_cfg* cfg, const qstate_stats* stats, uint8_t* widths_out,
                      uint32_t* head_off_out, void* stream) {
    int rc = validate(cfg);
    if (rc) return rc;
    if (!stats || !stats->ema_s || !stats->ema_r || !widths_out || !head_off_out ||
        (cfg->unit_kind == QSTATE_UNIT_ROW && !stats->range))
        return fail(QSTATE_EINVAL, "null pointer");
    int* status = nullptr;
    if ((rc = acquire_status(&status))) return rc;
    cudaError_t e;
    return run_alloc(cfg, stats->ema_s, stats->ema_r, stats->range, 0, widths_out, head_off_out,
                     status, static_cast<cudaStream_t>(stream));
}

int qstate_pack(const qstate_cfg* cfg, const float* S, qstate_buf* out, float* range_out, void* stream) {
    int rc = validate(cfg);
    if (rc) return rc;
    if (!S || !buf_ok(out)) return fail(QSTATE_EINVAL, "null pointer");
    int* status = nullptr;
    if ((rc = acquire_status(&status))) return rc;
    cudaError_t e;
    StepParams p = base_params(cfg, status);
    p.fit_every = 1;
    p.dense_in = S;
    p.out_payload = out->payload;
    p.out_scales = out->scales;
    p.out_widths = out->widths;
    p.out_head_off = out->head_off;
    p.out_fidx = out->fidx;
    p.range = range_out;
    e = launch_step_any(*cfg, 0, 1, p, static_cast<cudaStream_t>(stream));
    return e == cudaSuccess ? QSTATE_OK : cuda_fail(e, "pack kernel");
}

int qstate_unpack(const qstate_cfg* cfg, const qstate_buf* in, float* S_out, void* stream) {
    int rc = validate(cfg);
    if (rc) return rc;
    if (!S_out || !buf_ok(in)) return fail(QSTATE_EINVAL, "null pointer");
    int* status = nullptr;
    if ((rc = acquire_status(&status))) return rc;
    cudaError_t e;
    StepParams p = base_params(cfg, status);
    p.in_payload = in->payload;
    p.in_scales = in->scales;
    p.in_widths = in->widths;
    p.in_head_off = in->head_off;
    p.in_fidx = in->fidx;
    p.dense_out = S_out;
    e = launch_step_any(*cfg, 1, 0, p, static_cast<cudaStream_t>(stream));
    return e == cudaSuccess ? QSTATE_OK : cuda_fail(e, "unpack kernel");
}

int qstate_quant_decay(const qstate_cfg* cfg, const float* s, int32_t T, uint8_t* code_out,
                       float* lut_out, float* thr_out, void* stream) {
    int rc = validate(cfg);
    if (rc) return rc;
    if (cfg->gate_bits < 1) return fail(QSTATE_EINVAL, "gate_bits must be >= 1");
    if (!s || !code_out || !lut_out || !thr_out || T < 1) return fail(QSTATE_EINVAL, "null pointer or T < 1");
    int* status = nullptr;
    if ((rc = acquire_status(&status))) return rc;
    cudaError_t e;
    const int nchan = cfg->decay_kind == QSTATE_DECAY_ROW ? cfg->H * cfg->dk : cfg->H;
    const long long count = static_cast<long long>(cfg->B) * T;
    e = launch_quant_decay(s, count, nchan, cfg->gate_bits, code_out, lut_out, thr_out, status,
                           static_cast<cudaStream_t>(stream));
    return e == cudaSuccess ? QSTATE_OK : cuda_fail(e, "decay quantiser");
}

int qstate_quant_decay_noalloc(const qstate_cfg* cfg, const float* s, int32_t T, uint8_t* code_out,
                               float* lut_out, void* stream) {
    int rc = validate(cfg);
    if (rc) return rc;
    if (cfg->gate_bits < 1) return fail(QSTATE_EINVAL, "gate_bits must be >= 1");
    if (!s || !code_out || !lut_out || T < 1) return fail(QSTATE_EINVAL, "null pointer or T < 1");
    const int nchan = cfg->decay_kind == QSTATE_DECAY_ROW ? cfg->H * cfg->dk : cfg->H;
    const long long need = static_cast<long long>(nchan) * ((1 << cfg->gate_bits) - 1);
    if (need > quant_decay_scratch_capacity())
        return fail(QSTATE_EINVAL,
                    "qstate_quant_decay_noalloc: %lld thresholds (%d channels x %d) exceed the "
                    "built-in scratch of %lld; use qstate_quant_decay with a caller buffer",
                    need, nchan, (1 << cfg->gate_bits) - 1, quant_decay_scratch_capacity());
    int* status = nullptr;
    if ((rc = acquire_status(&status))) return rc;
    cudaError_t e;
    float* thr = nullptr;
    e = quant_decay_scratch(&thr);
    if (e != cudaSuccess) return cuda_fail(e, "threshold scratch lookup");
    const long long count = static_cast<long long>(cfg->B) * T;
    e = launch_quant_decay(s, count, nchan, cfg->gate_bits, code_out, lut_out, thr, status,
                           static_cast<cudaStream_t>(stream));
    return e == cudaSuccess ? QSTATE_OK : cuda_fail(e, "decay quantiser");
}

int qstate_step(const qstate_cfg* cfg, qstate_buf* in, qstate_buf* out, const qstate_inputs* x,
                int32_t t_begin, int32_t t_end, int32_t w_index, float* o, qstate_stats* stats,
                void* stream) {
    int rc = validate(cfg);
    if (rc) return rc;
    if (!buf_ok(in) || !buf_ok(out)) return fail(QSTATE_EINVAL, "null buffer pointer");
    if (!stats || !stats->ema_s || !stats->ema_r || (cfg->unit_kind == QSTATE_UNIT_ROW && !stats->range))
        return fail(QSTATE_EINVAL, "null statistics pointer");
    if ((rc = check_inputs(cfg, x, t_begin, t_end, o))) return rc;
    if (t_end - t_begin > cfg->C || t_end == t_begin)
        return fail(QSTATE_EINVAL, "a write-back interval holds 1..C tokens");
    if (x->s_code && cfg->gate_bits < 1) return fail(QSTATE_EINVAL, "s_code needs gate_bits");
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    int* status = nullptr;
    if ((rc = acquire_status(&status))) return rc;
    cudaError_t e;
    StepParams p = base_params(cfg, status);
    set_inputs(p, x);
    p.t_begin = t_begin;
    p.t_end = t_end;
    p.w_index = w_index;
    p.in_payload = in->payload;
    p.in_scales = in->scales;
    p.in_widths = in->widths;
    p.in_head_off = in->head_off;
    p.in_fidx = in->fidx;
    p.out_payload = out->payload;
    p.out_scales = out->scales;
    p.out_widths = out->widths;
    p.out_head_off = out->head_off;
    p.out_fidx = out->fidx;
    p.o = o;
    p.ema_s = stats->ema_s;
    p.ema_r = stats->ema_r;
    p.range = stats->range;
    if (cfg->alloc_mode == QSTATE_ALLOC_CURRENT) {
        // this write-back's statistics, the allocation from them, then the write-back proper
        if (!wb_row_eligible(*cfg, p))
            return fail(QSTATE_EINVAL, "alloc_mode current needs 16-byte aligned buffers and fidx");
        p.mode = 1;
        if ((e = launch_writeback(*cfg, p, st)) != cudaSuccess) return cuda_fail(e, "statistics pass");
        rc = run_alloc(cfg, stats->ema_s, stats->ema_r, stats->range, 0, out->widths,
                       out->head_off, status, st);
        if (rc) return rc;
        p.mode = 2;
        if ((e = launch_writeback(*cfg, p, st)) != cudaSuccess) return cuda_fail(e, "write-back kernel");
        return QSTATE_OK;
    }
    e = launch_writeback(*cfg, p, st);
    if (e != cudaSuccess) return cuda_fail(e, "write-back kernel");
    return run_alloc(cfg, stats->ema_s, stats->ema_r, stats->range, 0, in->widths, in->head_off,
                     status, st);
}

int qstate_scan(const qstate_cfg* cfg, qstate_buf* ping, qstate_buf* pong, const qstate_inputs* x,
                int32_t t_begin, int32_t t_end, int32_t w_index0, float* o, qstate_stats* stats,
                int32_t* final_in_pong, void* stream) {
    int rc = validate(cfg);
    if (rc) return rc;
    if ((rc = check_inputs(cfg, x, t_begin, t_end, o))) return rc;
    if (!buf_ok(ping) || !buf_ok(pong)) return fail(QSTATE_EINVAL, "null buffer pointer");
    if (!stats || !stats->ema_s || !stats->ema_r || (cfg->unit_kind == QSTATE_UNIT_ROW && !stats->range))
        return fail(QSTATE_EINVAL, "null statistics pointer");
    const int nsteps = t_end > t_begin ? (t_end - t_begin + cfg->C - 1) / cfg->C : 0;
    const int G = nsteps > 0 ? scan_parts(cfg, x, stats) : 1;
    if (G <= 1) {
        qstate_buf* src = ping;
        qstate_buf* dst = pong;
        int w = w_index0;
        for (int t0 = t_begin; t0 < t_end; t0 += cfg->C) {
            const int t1 = t0 + cfg->C < t_end ? t0 + cfg->C : t_end;
            rc = qstate_step(cfg, src, dst, x, t0, t1, w++, o, stats, stream);
            if (rc) return rc;
            qstate_buf* tmp = src;
            src = dst;
            dst = tmp;
        }
        if (final_in_pong) *final_in_pong = nsteps & 1;
        return QSTATE_OK;
    }
    // batch partitions [B p / G, B (p + 1) / G), one stream each (partition 0 on the caller's)
    int* status = nullptr;
    if ((rc = acquire_status(&status))) return rc;   // also makes the context current
    std::lock_guard<std::mutex> lock(g_part_mu);
    PartStreams* P = nullptr;
    if ((rc = part_streams(&P))) return rc;
    cudaStream_t cs = static_cast<cudaStream_t>(stream);
    qstate_cfg sub[kMaxParts];
    ScanArrays arr[kMaxParts];
    cudaStream_t ps[kMaxParts];
    for (int p = 0; p < G; ++p) {
        const long long b0 = static_cast<long long>(cfg->B) * p / G, b1 = static_cast<long long>(cfg->B) * (p + 1) / G;
        sub[p] = *cfg;
        sub[p].B = static_cast<int32_t>(b1 - b0);
        arr[p] = slice(cfg, ping, pong, x, o, stats, b0);
        ps[p] = p == 0 ? cs : P->s[p];
    }
    cudaError_t e = cudaEventRecord(P->fork, cs);
    for (int p = 1; p < G && e == cudaSuccess; ++p) e = cudaStreamWaitEvent(ps[p], P->fork, 0);
    if (e != cudaSuccess) return cuda_fail(e, "partition fork");
    int w = w_index0, flip = 0;
    for (int t0 = t_begin; t0 < t_end && rc == QSTATE_OK; t0 += cfg->C, ++w, flip ^= 1) {
        const int t1 = t0 + cfg->C < t_end ? t0 + cfg->C : t_end;
        for (int p = 0; p < G && rc == QSTATE_OK; ++p) {
            qstate_buf* src = flip ? &arr[p].pong : &arr[p].ping;
            qstate_buf* dst = flip ? &arr[p].ping : &arr[p].pong;
            rc = qstate_step(&sub[p], src, dst, &arr[p].x, t0, t1, w, arr[p].o, &arr[p].st, ps[p]);
        }
    }
    // join, also after a failed step, so that no partition's work is left unordered
    e = cudaSuccess;
    for (int p = 1; p < G; ++p) {
        cudaError_t e1 = cudaEventRecord(P->join[p], ps[p]);
        if (e1 == cudaSuccess) e1 = cudaStreamWaitEvent(cs, P->join[p], 0);
        if (e == cudaSuccess) e = e1;
    }
    if (rc) return rc;
    if (e != cudaSuccess) return cuda_fail(e, "partition join");
    if (final_in_pong) *final_in_pong = nsteps & 1;
    return QSTATE_OK;
}

int qstate_scan_partition_count(const qstate_cfg* cfg, const qstate_inputs* x, const qstate_stats* stats) {
    if (validate(cfg) != QSTATE_OK || !x || !x->q || !x->k || !x->v || !stats || !stats->ema_s || !stats->ema_r)
        return 0;
    return scan_parts(cfg, x, stats);
}

int qstate_set_scan_partitions(int32_t n) {
    if (n < 0 || n > kMaxParts) return fail(QSTATE_EINVAL, "partitions must be in [0, %d]", kMaxParts);
    g_scan_parts.store(n);
    return QSTATE_OK;
}

int qstate_scan_host(const qstate_cfg* cfg, qstate_buf* ping, qstate_buf* pong,
                     const qstate_inputs* x_host, const qstate_inputs* x_dev, int32_t t_begin,
                     int32_t t_end, int32_t w_index0, float* o_host, float* o_dev,
                     qstate_stats* stats, int32_t chunk, int32_t* final_in_pong, void* stream,
                     void* copy_stream) {
    int rc = validate(cfg);
    if (rc) return rc;
    if ((rc = check_inputs(cfg, x_dev, t_begin, t_end, o_dev))) return rc;
    if (!x_host || !o_host || x_host->T != x_dev->T)
        return fail(QSTATE_EINVAL, "host inputs / readouts missing or of another length");
    if (!stream || !copy_stream || stream == copy_stream)
        return fail(QSTATE_EINVAL, "need two distinct non-default streams");
    if (chunk < 1 || chunk % cfg->C != 0) return fail(QSTATE_EINVAL, "chunk must be a multiple of C");
    // every input given on the host side must have a device buffer to land in
    const bool bad = (x_host->q && !x_dev->q) || (x_host->k && !x_dev->k) || (x_host->v && !x_dev->v) ||
                     (x_host->beta && !x_dev->beta) || (x_host->s && !x_dev->s) ||
                     (x_host->s_code && !x_dev->s_code) || (x_host->a && !x_dev->a) ||
                     (x_host->w && !x_dev->w);
    if (bad) return fail(QSTATE_EINVAL, "a host input has no device buffer");
    cudaStream_t cs = static_cast<cudaStream_t>(stream), ts = static_cast<cudaStream_t>(copy_stream);
    // readouts go back on a library-owned stream, so that they move while later chunks'
    // inputs come in (the host link carries both directions at once)
    cudaStream_t rs = nullptr;
    {
        int* status = nullptr;
        if ((rc = acquire_status(&status))) return rc;   // also makes the context current
        std::lock_guard<std::mutex> lock(g_part_mu);
        PartStreams* P = nullptr;
        if ((rc = part_streams(&P))) return rc;
        rs = P->rd;
    }
    const int B = cfg->B, T = x_dev->T, H = cfg->H;
    const size_t f4 = sizeof(float);
    const size_t nchan = cfg->decay_kind == QSTATE_DECAY_ROW ? static_cast<size_t>(H) * cfg->dk : H;
    struct Item { void* d; const void* h; size_t per; };
    const Item in[8] = {{(void*)x_dev->q, x_host->q, H * cfg->dk * f4}, {(void*)x_dev->k, x_host->k, H * cfg->dk * f4},
                        {(void*)x_dev->v, x_host->v, H * cfg->dv * f4}, {(void*)x_dev->beta, x_host->beta, H * f4},
                        {(void*)x_dev->s, x_host->s, nchan * f4}, {(void*)x_dev->s_code, x_host->s_code, nchan},
                        {(void*)x_dev->a, x_host->a, H * cfg->dk * f4}, {(void*)x_dev->w, x_host->w, H * cfg->dv * f4}};
    // tokens [t0, t1) of a (B, T, per) token-major tensor: one copy per batch element (one
    // copy in all when the chunk spans every token); plain copies move pinned host memory at
    // full link speed where strided 2D copies were measured several times slower
    auto copy_tokens = [&](void* dst, const void* src, size_t per, int t0, int t1, cudaMemcpyKind kind,
                           cudaStream_t cst) {
        const size_t pitch = static_cast<size_t>(T) * per, off = static_cast<size_t>(t0) * per;
        const size_t width = static_cast<size_t>(t1 - t0) * per;
        if (width == pitch)
            return cudaMemcpyAsync(dst, src, pitch * B, kind, cst);
        const bool a16 = per % 16 == 0 && (reinterpret_cast<uintptr_t>(dst) & 15) == 0 &&
                         (reinterpret_cast<uintptr_t>(src) & 15) == 0;
        if (a16) {
            stage_tokens_kernel<<<2 * device_sm_count(), 128, 0, cst>>>(static_cast<uint4*>(dst), static_cast<const uint4*>(src),
                                                        B, static_cast<long long>(pitch / 16),
                                                        static_cast<long long>(off / 16),
                                                        static_cast<long long>(width / 16));
            return cudaGetLastError();
        }
        cudaError_t err = cudaSuccess;
        for (int bb = 0; bb < B && err == cudaSuccess; ++bb)
            err = cudaMemcpyAsync(static_cast<char*>(dst) + bb * pitch + off,
                                  static_cast<const char*>(src) + bb * pitch + off, width, kind, cst);
        return err;
    };
    qstate_buf* src = ping;
    qstate_buf* dst = pong;
    int in_pong = 0, w = w_index0;
    cudaError_t e = cudaSuccess;
    cudaEvent_t ev_in = nullptr, ev_out = nullptr;
    // Inputs of chunk c + 1 are queued on the copy stream once chunk c's scan is queued, so they
    // move while chunk c computes (they fill other tokens of the device buffers); the readouts of
    // chunk c follow on the readout stream once it is done.
    auto stage_inputs = [&](int c0, int c1) {
        for (const Item& it : in)
            if (it.h && e == cudaSuccess) e = copy_tokens(it.d, it.h, it.per, c0, c1, cudaMemcpyHostToDevice, ts);
        if (e == cudaSuccess) e = cudaEventCreateWithFlags(&ev_in, cudaEventDisableTiming);
        if (e == cudaSuccess) e = cudaEventRecord(ev_in, ts);
    };
    if (t_begin < t_end) stage_inputs(t_begin, t_begin + chunk < t_end ? t_begin + chunk : t_end);
    for (int c0 = t_begin; c0 < t_end && e == cudaSuccess && rc == QSTATE_OK; c0 += chunk) {
        const int c1 = c0 + chunk < t_end ? c0 + chunk : t_end;
        e = cudaStreamWaitEvent(cs, ev_in, 0);
        cudaEventDestroy(ev_in);
        ev_in = nullptr;
        if (e != cudaSuccess) break;
        int flip = 0;
        rc = qstate_scan(cfg, src, dst, x_dev, c0, c1, w, o_dev, stats, &flip, stream);
        if (rc) break;
        w += (c1 - c0 + cfg->C - 1) / cfg->C;
        if (flip) {
            qstate_buf* tmp = src;
            src = dst;
            dst = tmp;
            in_pong ^= 1;
        }
        if (c1 < t_end) stage_inputs(c1, c1 + chunk < t_end ? c1 + chunk : t_end);
        if (e == cudaSuccess) e = cudaEventCreateWithFlags(&ev_out, cudaEventDisableTiming);
        if (e == cudaSuccess) e = cudaEventRecord(ev_out, cs);
        if (e == cudaSuccess) e = cudaStreamWaitEvent(rs, ev_out, 0);
        if (ev_out) cudaEventDestroy(ev_out);
        ev_out = nullptr;
        if (e == cudaSuccess) e = copy_tokens(o_host, o_dev, H * cfg->dv * f4, c0, c1, cudaMemcpyDeviceToHost, rs);
    }
    if (ev_in) cudaEventDestroy(ev_in);
    // the compute stream completes only after the last readout copy (also after a failure, so
    // that no copy on the library's stream is left unordered)
    {
        cudaError_t e1 = cudaEventCreateWithFlags(&ev_out, cudaEventDisableTiming);
        if (e1 == cudaSuccess) e1 = cudaEventRecord(ev_out, rs);
        if (e1 == cudaSuccess) e1 = cudaStreamWaitEvent(cs, ev_out, 0);
        if (ev_out) cudaEventDestroy(ev_out);
        if (e == cudaSuccess) e = e1;
    }
    if (rc) return rc;
    if (e != cudaSuccess) return cuda_fail(e, "host staging");
    if (final_in_pong) *final_in_pong = in_pong;
    return QSTATE_OK;
}

int qstate_scan_fp32(const qstate_cfg* cfg, float* S, const qstate_inputs* x, int32_t t_begin,
                     int32_t t_end, float* o, void* stream) {
    int rc = validate(cfg);
    if (rc) return rc;
    if (!S) return fail(QSTATE_EINVAL, "S is NULL");
    if ((rc = check_inputs(cfg, x, t_begin, t_end, o))) return rc;
    int* status = nullptr;
    if ((rc = acquire_status(&status))) return rc;
    cudaError_t e;
    StepParams p = base_params(cfg, status);
    set_inputs(p, x);
    p.dense_in = S;
    p.dense_out = S;
    p.o = o;
    for (int t0 = t_begin; t0 < t_end; t0 += cfg->C) {
        p.t_begin = t0;
        p.t_end = t0 + cfg->C < t_end ? t0 + cfg->C : t_end;
        e = launch_step_any(*cfg, 0, 0, p, static_cast<cudaStream_t>(stream));
        if (e != cudaSuccess) return cuda_fail(e, "fp32 write-back kernel");
    }
    return QSTATE_OK;
}

int qstate_check(void* stream) {
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    cudaError_t e = cudaStreamSynchronize(st);
    if (e != cudaSuccess) return cuda_fail(e, "stream synchronize");
    int dev = -1;
    int* status = status_word(&e, &dev);
    if (!status) return cuda_fail(e, "status word");
    int v = 0;
    e = cudaMemcpy(&v, status, sizeof(int), cudaMemcpyDeviceToHost);
    if (e != cudaSuccess) return cuda_fail(e, "status read");
    if (v != 0) {
        const int zero = 0;
        e = cudaMemcpy(status, &zero, sizeof(int), cudaMemcpyHostToDevice);
        if (e != cudaSuccess) return cuda_fail(e, "status clear");
        if (v & QS_DEV_TEARDOWN) g_unusable[dev].store(true);
        const int code = (v & QS_DEV_TEARDOWN) ? QSTATE_EDEVICE
                         : (v & QS_DEV_TIMEOUT) ? QSTATE_ETIMEOUT : QSTATE_EDEVICE;
        return fail(code, "device status 0x%x:%s%s%s%s%s", v,
                    (v & QS_DEV_LAYOUT) ? " inconsistent widths/offsets" : "",
                    (v & QS_DEV_RATE) ? " decay rate not positive/finite" : "",
                    (v & QS_DEV_TIMEOUT) ? " tensor-core product timed out" : "",
                    (v & QS_DEV_CHUNK) ? " decay over a 16-token block beyond the chunked form's range" : "",
                    (v & QS_DEV_TEARDOWN) ? " the wait before freeing tensor memory gave up too: device marked unusable" : "");
    }
    if (g_unusable[dev].load())
        return fail(QSTATE_EDEVICE, "device %d is marked unusable: a tensor-core teardown wait gave up "
                    "earlier in this process", dev);
    return QSTATE_OK;
}

int qstate_set_wait_limit(int32_t polls) {
    g_wait_polls.store(polls < 0 ? kDefaultWaitPolls : polls);
    return QSTATE_OK;
}

const char* qstate_last_error(void) { return g_err; }

}  // extern "C"
