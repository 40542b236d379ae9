/*
 * qstate_oracle.c -- plain, slow CPU reference of the low-bit recurrent-state method of
 * "Low-Bit Recurrent States in Hybrid Language Models" (Chen & He, 2026).
 *
 * TEST INFRASTRUCTURE ONLY.  The test-suite, the smoke check and the benchmark's CPU
 * baseline load this file; the product library never links, loads or calls it, and the two
 * share no code, header, table or constant.  Build: gcc -O2 -ffp-contract=off (no FMA
 * contraction, no fast-math), so every float operation below is one IEEE-rounded operation.
 *
 * Precision.  The paper keeps recurrent states in FP32 (Sec. 1, Sec. 4 "FP32 states"), so
 * the state arithmetic here is FP32; an FP64 recurrence is given alongside as the exact
 * reference.  Where floating point decides an integer -- a quantised code, the fitted range
 * factor, a bit width, a log-decay code -- the decision is taken in FP32 with the operation
 * sequence documented at each function, which is the precision the kernels decide in.
 *
 * Parity unpinned: none.  Every function here is pinned by a CPU test against closed forms,
 * printed values of the paper, brute force or an independent formulation.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

/* ---------------------------------------------------------------------------------------
 * Configuration (mirrored by oracle/oracle.py; unrelated to the library's own struct).
 * ------------------------------------------------------------------------------------- */
typedef struct {
    int32_t B, H, dk, dv;
    int32_t decay_kind;  /* 0: rate per row (KDA); 1: rate per head (Gated DeltaNet, Mamba-2) */
    int32_t erase_kind;  /* 0: a = beta k, w = beta 1 (KDA, GDN); 1: a = 0, w = 1 (Mamba-2)   */
    int32_t unit_kind;   /* 0: width + FP16 scale per row; 1: width per head, scale per 32 rows x column */
    int32_t group_heads; /* heads per output-normalisation group u(i) (row unit)               */
    int32_t bbar_num, bbar_den; /* mean payload bits per element, as a fraction            */
    int32_t bmin, bmax;
    int32_t C;           /* write-back period in tokens                                       */
    int32_t fit_every;   /* 1: fit the range factor at every write-back                      */
    float ema_span;      /* 64 tokens                                                         */
    int32_t gate_bits;   /* 0: FP32 rates; g > 0: log-quantised rates                         */
    int32_t weight_kind; /* 0: c = Gamma_hat * Rtilde^2 (Eq. 3)                                */
    int32_t alloc_mode;  /* 0: widths from the previous write-back's statistics (lagged);
                            1: widths from this write-back's statistics (orc_step_current)  */
} orc_cfg;

#define ORC_OK 0
#define ORC_EINVAL 1
#define ORC_EBUDGET 2
#define NFIT 16

/* ---------------------------------------------------------------------------------------
 * Small helpers.
 * ------------------------------------------------------------------------------------- */

/* IEEE binary16, round to nearest even, magnitudes saturated at 65504 (Sec. 3, "Levels and
 * storage": the fitted scale is stored as FP16). */
static uint16_t f16_bits(float x) {
    if (x > 65504.0f) x = 65504.0f;
    if (x < -65504.0f) x = -65504.0f;
    _Float16 h = (_Float16)x;
    uint16_t u;
    memcpy(&u, &h, 2);
    return u;
}

static float f16_value(uint16_t u) {
    _Float16 h;
    memcpy(&h, &u, 2);
    return (float)h;
}

/* The 16 candidate range factors in [1/4, 1] (Sec. 3, "Levels and storage"): evenly spaced,
 * both ends included: f_k = (5 + k) / 20, rounded to FP32. */
static float fit_factor(int k) { return (float)((5.0 + (double)k) / 20.0); }

/* expm1 in FP32 from its Taylor series (degree 16, Horner order, one rounding per operation),
 * with expm1(2y) = expm1(y) (expm1(y) + 2) applied while the argument exceeds 1.  The
 * coefficients are 1/k! computed in FP64 and rounded to FP32.  Used by the allocation weight
 * (Eq. 3) so that widths are reproducible bit for bit; defined for x >= 0 (0 below). */
float orc_expm1_series(float x) {
    if (!(x > 0.0f)) return 0.0f;
    int halvings = 0;
    while (x > 1.0f) {
        x = x * 0.5f;
        halvings++;
    }
    float c[17];
    double fact = 1.0;
    for (int k = 1; k <= 16; k++) {
        fact *= (double)k;
        c[k] = (float)(1.0 / fact);
    }
    float p = c[16];
    for (int k = 15; k >= 1; k--) p = p * x + c[k];
    float y = p * x;
    for (int i = 0; i < halvings; i++) y = y * (y + 2.0f);
    return y;
}

double orc_bits_per_element(const orc_cfg* c) {
    /* Sec. 3, "Levels and storage": FP16 scale + width bits per row element; block scales
     * add 16/32 = 0.5 bit; per-head widths are counted too. */
    double bbar = (double)c->bbar_num / (double)c->bbar_den;
    int levels = c->bmax - c->bmin + 1, wbits = 0;
    while ((1 << wbits) < levels) wbits++;
    if (c->unit_kind == 0) return bbar + (16.0 + wbits) / (double)c->dv;
    return bbar + 16.0 / 32.0 + (double)wbits / ((double)c->dk * (double)c->dv);
}

/* ---------------------------------------------------------------------------------------
 * Eq. (1): S_t = (I - k a^T) D_t S_{t-1} + k (w o v)^T,  o_t = S_t^T q_t,  D_t = diag(e^{-s}).
 * Unquantised, one head, T tokens.  S is dk x dv, row-major (rows = key channels, on which
 * the decay acts; columns = value channels).  Per token t: k, q, a, s are dk-vectors, v, w
 * dv-vectors.  o receives T x dv readouts.
 * ------------------------------------------------------------------------------------- */
void orc_recur_f32(int dk, int dv, int T, float* S, const float* k, const float* q,
                   const float* v, const float* s, const float* a, const float* w, float* o) {
    float* y = (float*)malloc(sizeof(float) * dv);
    for (int t = 0; t < T; t++) {
        const float *kt = k + (size_t)t * dk, *qt = q + (size_t)t * dk, *at = a + (size_t)t * dk;
        const float *st = s + (size_t)t * dk, *vt = v + (size_t)t * dv, *wt = w + (size_t)t * dv;
        for (int i = 0; i < dk; i++) {           /* S' = D_t S */
            float d = expf(-st[i]);
            for (int j = 0; j < dv; j++) S[i * dv + j] = S[i * dv + j] * d;
        }
        for (int j = 0; j < dv; j++) {           /* y = a^T S' */
            float acc = 0.0f;
            for (int i = 0; i < dk; i++) acc = acc + at[i] * S[i * dv + j];
            y[j] = acc;
        }
        for (int i = 0; i < dk; i++)             /* S = S' - k y^T + k (w o v)^T */
            for (int j = 0; j < dv; j++)
                S[i * dv + j] = (S[i * dv + j] - kt[i] * y[j]) + kt[i] * (wt[j] * vt[j]);
        for (int j = 0; j < dv; j++) {           /* o = S^T q */
            float acc = 0.0f;
            for (int i = 0; i < dk; i++) acc = acc + S[i * dv + j] * qt[i];
            o[(size_t)t * dv + j] = acc;
        }
    }
    free(y);
}

void orc_recur_f64(int dk, int dv, int T, double* S, const float* k, const float* q,
                   const float* v, const float* s, const float* a, const float* w, double* o) {
    double* y = (double*)malloc(sizeof(double) * dv);
    for (int t = 0; t < T; t++) {
        const float *kt = k + (size_t)t * dk, *qt = q + (size_t)t * dk, *at = a + (size_t)t * dk;
        const float *st = s + (size_t)t * dk, *vt = v + (size_t)t * dv, *wt = w + (size_t)t * dv;
        for (int i = 0; i < dk; i++) {
            double d = exp(-(double)st[i]);
            for (int j = 0; j < dv; j++) S[i * dv + j] *= d;
        }
        for (int j = 0; j < dv; j++) {
            double acc = 0.0;
            for (int i = 0; i < dk; i++) acc += (double)at[i] * S[i * dv + j];
            y[j] = acc;
        }
        for (int i = 0; i < dk; i++)
            for (int j = 0; j < dv; j++)
                S[i * dv + j] += -(double)kt[i] * y[j] + (double)kt[i] * ((double)wt[j] * vt[j]);
        for (int j = 0; j < dv; j++) {
            double acc = 0.0;
            for (int i = 0; i < dk; i++) acc += S[i * dv + j] * (double)qt[i];
            o[(size_t)t * dv + j] = acc;
        }
    }
    free(y);
}

/* ---------------------------------------------------------------------------------------
 * Sec. 3, "Levels and storage": quantise one scale group x[0], x[stride], ... (g elements)
 * to b bits.
 *   b = 0: nothing is stored; the group dequantises to zero.
 *   b = 1: sign times mean absolute value: m = FP16((sum |x|) / g); code 1 for x < 0.
 *   b >= 2: levels {-n..n} Delta, n = 2^(b-1) - 1, Delta = f R / n, R = max |x|, f fitted
 *           over 16 values in [1/4, 1] by the group's squared error; Delta stored as FP16.
 * Operation sequence (FP32, one rounding each):
 *   Delta_k = FP16(FP32(f_k * R) * FP32(1/n)),  inv_k = 1 / Delta_k (0 if Delta_k = 0),
 *   q = clamp(rint(x * inv_k), -n, n),  e = x - q * Delta_k,  SSE_k = sum e^2 (in index order).
 * The smallest SSE wins; equal SSEs go to the larger f (so R = 0 gives f = 1).  Codes are
 * offset binary u = q + n.  refit = 0 reuses factor fidx_in instead of searching; widths 0
 * and 1 do not use a factor and carry fidx_in over unchanged.  sse16 (optional) receives every
 * candidate's SSE recomputed in FP64 from the same codes, for near-tie checks.
 * ------------------------------------------------------------------------------------- */
void orc_quant_group(const float* x, int g, int stride, int b, int refit, int fidx_in,
                     uint16_t* codes, uint16_t* scale, uint8_t* fidx, double* sse16) {
    if (b <= 0) {
        *scale = 0;
        *fidx = (uint8_t)fidx_in;
        return;
    }
    if (b == 1) {
        float acc = 0.0f;
        for (int j = 0; j < g; j++) acc = acc + fabsf(x[(size_t)j * stride]);
        float m = acc / (float)g;
        *scale = f16_bits(m);
        *fidx = (uint8_t)fidx_in;
        for (int j = 0; j < g; j++) codes[j] = (x[(size_t)j * stride] < 0.0f) ? 1 : 0;
        return;
    }
    int n = (1 << (b - 1)) - 1;
    float R = 0.0f;
    for (int j = 0; j < g; j++) {
        float a = fabsf(x[(size_t)j * stride]);
        if (a > R) R = a;
    }
    if (sse16)
        for (int k = 0; k < NFIT; k++) sse16[k] = 0.0;
    if (R == 0.0f) {
        *scale = 0;
        *fidx = (uint8_t)(refit ? NFIT - 1 : fidx_in);
        for (int j = 0; j < g; j++) codes[j] = (uint16_t)n;
        return;
    }
    float inv_n = 1.0f / (float)n;
    int best = -1;
    float best_sse = 0.0f;
    int klo = refit ? 0 : fidx_in, khi = refit ? NFIT - 1 : fidx_in;
    for (int k = khi; k >= klo; k--) {
        float fr = fit_factor(k) * R;
        uint16_t dh = f16_bits(fr * inv_n);
        float D = f16_value(dh);
        float inv = (D == 0.0f) ? 0.0f : 1.0f / D;
        float sse = 0.0f;
        double sse64 = 0.0;
        for (int j = 0; j < g; j++) {
            float xj = x[(size_t)j * stride];
            float qf = rintf(xj * inv);
            if (qf > (float)n) qf = (float)n;
            if (qf < (float)-n) qf = (float)-n;
            float e = xj - qf * D;
            sse = sse + e * e;
            double e64 = (double)xj - (double)qf * (double)D;
            sse64 += e64 * e64;
        }
        if (sse16) sse16[k] = sse64;
        if (best < 0 || sse < best_sse) {
            best = k;
            best_sse = sse;
        }
    }
    float D = f16_value(f16_bits((fit_factor(best) * R) * inv_n));
    float inv = (D == 0.0f) ? 0.0f : 1.0f / D;
    *scale = f16_bits((fit_factor(best) * R) * inv_n);
    *fidx = (uint8_t)best;
    for (int j = 0; j < g; j++) {
        float qf = rintf(x[(size_t)j * stride] * inv);
        if (qf > (float)n) qf = (float)n;
        if (qf < (float)-n) qf = (float)-n;
        codes[j] = (uint16_t)((int)qf + n);
    }
}

/* Inverse of the levels: b = 0 -> 0; b = 1 -> +-m; b >= 2 -> (u - n) * Delta (FP32). */
void orc_dequant_group(const uint16_t* codes, int g, int b, uint16_t scale, float* x, int stride) {
    float D = f16_value(scale);
    int n = (b >= 2) ? (1 << (b - 1)) - 1 : 0;
    for (int j = 0; j < g; j++) {
        float val;
        if (b <= 0) val = 0.0f;
        else if (b == 1) val = codes[j] ? -D : D;
        else val = (float)((int)codes[j] - n) * D;
        x[(size_t)j * stride] = val;
    }
}

/* Bit layout of one row: element j's b-bit code occupies bits [j b, j b + b) of the row,
 * bit m of the row being bit (m mod 8) of byte m / 8 (least significant first).  A row of
 * dv elements takes exactly b dv / 8 bytes: no padding, no ternary packing (Sec. 3). */
void orc_pack_codes(const uint16_t* codes, int g, int b, uint8_t* dst) {
    memset(dst, 0, (size_t)b * g / 8);
    for (int j = 0; j < g; j++)
        for (int p = 0; p < b; p++)
            if ((codes[j] >> p) & 1) {
                long m = (long)j * b + p;
                dst[m / 8] |= (uint8_t)(1u << (m % 8));
            }
}

void orc_unpack_codes(const uint8_t* src, int g, int b, uint16_t* codes) {
    for (int j = 0; j < g; j++) {
        unsigned u = 0;
        for (int p = 0; p < b; p++) {
            long m = (long)j * b + p;
            u |= (unsigned)((src[m / 8] >> (m % 8)) & 1) << p;
        }
        codes[j] = (uint16_t)u;
    }
}

/* ---------------------------------------------------------------------------------------
 * State layout.  Batch element b owns one payload region of exactly H dk dv bbar / 8 bytes
 * (the layer-wise budget).  Inside it, heads h = 0..H-1 follow each other, rows i = 0..dk-1
 * inside a head; head h starts at byte head_off[b H + h] and row i at the prefix sum of the
 * widths of rows 0..i-1 (Sec. 3: "Prefix sums of widths give row offsets").
 * ------------------------------------------------------------------------------------- */
long orc_region_bytes(const orc_cfg* c) {
    long bits = (long)c->H * c->dk * c->dv * c->bbar_num;
    if (bits % ((long)8 * c->bbar_den)) return -1;
    return bits / (8L * c->bbar_den);
}

static int unit_width(const orc_cfg* c, const uint8_t* widths, int b, int h, int i) {
    if (c->unit_kind == 0) return widths[((size_t)b * c->H + h) * c->dk + i];
    return widths[(size_t)b * c->H + h];
}

static long row_offset(const orc_cfg* c, const uint8_t* widths, const uint32_t* head_off, int b,
                       int h, int i) {
    long off = (long)b * orc_region_bytes(c) + head_off[(size_t)b * c->H + h];
    for (int r = 0; r < i; r++) off += (long)unit_width(c, widths, b, h, r) * c->dv / 8;
    return off;
}

/* Scale group g of head (b, h): row unit -> row i (dv elements, stride 1); head unit ->
 * block of 32 key rows x one value column (32 elements, stride dv). */
static size_t scale_index(const orc_cfg* c, int b, int h, int i, int j) {
    if (c->unit_kind == 0) return ((size_t)b * c->H + h) * c->dk + i;
    return (((size_t)b * c->H + h) * (c->dk / 32) + i / 32) * c->dv + j;
}

/* A width map and head offsets describe a valid layout when every width lies in [0, 16],
 * heads follow each other without overlap and the last head ends inside the region. */
static int layout_ok(const orc_cfg* c, const uint8_t* widths, const uint32_t* head_off) {
    long rb = orc_region_bytes(c);
    if (rb < 0) return 0;
    for (int b = 0; b < c->B; b++) {
        long end = 0;
        for (int h = 0; h < c->H; h++) {
            if ((long)head_off[(size_t)b * c->H + h] < end) return 0;
            long bytes = 0;
            for (int i = 0; i < c->dk; i++) {
                int bw = unit_width(c, widths, b, h, i);
                if (bw < 0 || bw > 16) return 0;
                bytes += (long)bw * c->dv / 8;
            }
            end = (long)head_off[(size_t)b * c->H + h] + bytes;
        }
        if (end > rb) return 0;
    }
    return 1;
}

/* Quantise + pack one head's dense FP32 state X (dk x dv) with the widths of the target
 * buffer (Sec. 3).  Row unit: R_i (the row absmax) is written to range[row]. */
static void pack_head(const orc_cfg* c, int b, int h, const float* X, const uint8_t* widths,
                      const uint32_t* head_off, int refit, const uint8_t* fidx_in,
                      uint8_t* payload, uint16_t* scales, uint8_t* fidx_out, float* range) {
    int dk = c->dk, dv = c->dv;
    uint16_t* codes = (uint16_t*)malloc(sizeof(uint16_t) * (size_t)dk * dv);
    if (c->unit_kind == 0) {
        for (int i = 0; i < dk; i++) {
            int bw = unit_width(c, widths, b, h, i);
            size_t si = scale_index(c, b, h, i, 0);
            const float* row = X + (size_t)i * dv;
            float R = 0.0f;
            for (int j = 0; j < dv; j++)
                if (fabsf(row[j]) > R) R = fabsf(row[j]);
            if (range) range[((size_t)b * c->H + h) * dk + i] = R;
            int fin = fidx_in ? fidx_in[si] : NFIT - 1;
            orc_quant_group(row, dv, 1, bw, refit, fin, codes + (size_t)i * dv, &scales[si],
                            &fidx_out[si], NULL);
        }
    } else {
        int bw = unit_width(c, widths, b, h, 0);
        for (int blk = 0; blk < dk / 32; blk++)
            for (int j = 0; j < dv; j++) {
                size_t si = scale_index(c, b, h, blk * 32, j);
                uint16_t cc[32];
                int fin = fidx_in ? fidx_in[si] : NFIT - 1;
                orc_quant_group(X + (size_t)blk * 32 * dv + j, 32, dv, bw, refit, fin, cc,
                                &scales[si], &fidx_out[si], NULL);
                for (int r = 0; r < 32; r++) codes[(size_t)(blk * 32 + r) * dv + j] = cc[r];
            }
    }
    for (int i = 0; i < dk; i++) {
        int bw = unit_width(c, widths, b, h, i);
        if (bw > 0)
            orc_pack_codes(codes + (size_t)i * dv, dv, bw,
                           payload + row_offset(c, widths, head_off, b, h, i));
    }
    free(codes);
}

static void unpack_head(const orc_cfg* c, int b, int h, const uint8_t* payload,
                        const uint16_t* scales, const uint8_t* widths, const uint32_t* head_off,
                        float* X) {
    int dk = c->dk, dv = c->dv;
    uint16_t* codes = (uint16_t*)malloc(sizeof(uint16_t) * (size_t)dv);
    for (int i = 0; i < dk; i++) {
        int bw = unit_width(c, widths, b, h, i);
        if (bw > 0)
            orc_unpack_codes(payload + row_offset(c, widths, head_off, b, h, i), dv, bw, codes);
        else
            memset(codes, 0, sizeof(uint16_t) * dv);
        if (c->unit_kind == 0) {
            orc_dequant_group(codes, dv, bw, scales[scale_index(c, b, h, i, 0)],
                              X + (size_t)i * dv, 1);
        } else {
            for (int j = 0; j < dv; j++)
                orc_dequant_group(codes + j, 1, bw, scales[scale_index(c, b, h, i, j)],
                                  X + (size_t)i * dv + j, 1);
        }
    }
    free(codes);
}

/* Whole-state quantise + pack of a dense state S (B, H, dk, dv), always fitting f. */
int orc_pack(const orc_cfg* c, const float* S, const uint8_t* widths, const uint32_t* head_off,
             uint8_t* payload, uint16_t* scales, uint8_t* fidx, float* range) {
    long rb = orc_region_bytes(c);
    if (rb < 0 || !layout_ok(c, widths, head_off)) return ORC_EINVAL;
    memset(payload, 0, (size_t)rb * c->B);
    for (int b = 0; b < c->B; b++)
        for (int h = 0; h < c->H; h++)
            pack_head(c, b, h, S + ((size_t)b * c->H + h) * c->dk * c->dv, widths, head_off, 1,
                      NULL, payload, scales, fidx, range);
    return ORC_OK;
}

int orc_unpack(const orc_cfg* c, const uint8_t* payload, const uint16_t* scales,
               const uint8_t* widths, const uint32_t* head_off, float* S) {
    if (!layout_ok(c, widths, head_off)) return ORC_EINVAL;
    for (int b = 0; b < c->B; b++)
        for (int h = 0; h < c->H; h++)
            unpack_head(c, b, h, payload, scales, widths, head_off,
                        S + ((size_t)b * c->H + h) * c->dk * c->dv);
    return ORC_OK;
}

/* ---------------------------------------------------------------------------------------
 * Sec. 3, "State bit allocation".
 *
 * Eq. (3): c_i = Gamma_hat_i Rtilde_i^2,  Gamma_hat_i = 1 / expm1(2 (s_hat_i + r_i)),
 *   s_hat_i = -1/2 log EMA(e^{-2 s}),  r_i = 1/2 EMA[beta (2 - beta) k_i^2].
 * With m_s = EMA(1 - e^{-2s}) (the complement is kept because EMA is linear and it stays
 * accurate for slowly decaying rows) and m_r = EMA[beta (2 - beta) k_i^2]:
 *   2 (s_hat + r) = -log(1 - m_s) + m_r  =>  Gamma_hat = (1 - m_s) / (expm1(m_r) + m_s).
 * Rtilde_i^2 = R_i^2 / mean_{j in u(i)} R_j^2 (RMS over the output-normalisation group, the
 * sum taken in row order); 1 when that mean is 0.  The head unit uses Rtilde = 1.
 * FP32 sequence: G = (1 - m_s) / (expm1(max(m_r, 0)) + m_s); c = G * (R * R / mean).
 * Weights below 2^-60 (and NaN) become the null weight 2^-200; weights above 2^60 are
 * clamped to 2^60.
 * ------------------------------------------------------------------------------------- */
/* Table 1 replaces c_i by other weights; weight_kind selects one (0 is Eq. 3):
 *   1  R^2                     range alone
 *   2  Gamma_hat R^2           raw range
 *   3  Rtilde^2                relative range
 *   4  w1 Rtilde^2             persistence w1 = 1/(1 - e^{-2 s_hat}) = 1/m_s
 *   5  h Rtilde^2              write-back factor h = 1/(1 - e^{-2 C s_hat}) = 1/(1 - (1 - m_s)^C),
 *                              the power by repeated squaring (low bit of C first)
 *   6  Gamma_hat(m_r = 0) Rtilde^2   erasure left out
 *   7  Gamma_hat_{pi(i)} Rtilde_i^2  decay weights moved to other units by the bijection
 *                              pi(i) = (A i + N/3) mod N, A the smallest integer > 0.6180339887 N
 *                              coprime to N (N units per batch element)
 *   8  1                        uniform widths
 * The head unit has no per-unit range: R = Rtilde = 1 there. */
static int orc_gcd(int a, int b) { return b == 0 ? a : orc_gcd(b, a % b); }

void orc_shuffle(int N, int* A, int* B0) {
    int a = (int)(0.6180339887 * N) + 1;
    while (orc_gcd(a, N) != 1) a++;
    *A = a % N;
    *B0 = N / 3;
}

static float weight_of(const orc_cfg* c, int kind, float ms, float mr, float R2, float rt2) {
    if (kind == 1) return R2;
    if (kind == 3) return rt2;
    if (kind == 8) return 1.0f;
    if (kind == 4) return (1.0f / ms) * rt2;
    if (kind == 5) {
        float pw = 1.0f, bb = 1.0f - ms;
        for (int e = c->C; e > 0; e >>= 1) {
            if (e & 1) pw = pw * bb;
            bb = bb * bb;
        }
        return (1.0f / (1.0f - pw)) * rt2;
    }
    if (kind == 6) mr = 0.0f;
    if (mr < 0.0f) mr = 0.0f;
    float G = (1.0f - ms) / (orc_expm1_series(mr) + ms);
    if (kind == 2) return G * R2;
    return G * rt2;   /* 0, 6, 7 */
}

int orc_weights(const orc_cfg* c, int b, const float* ema_s, const float* ema_r,
                const float* range, float* cw) {
    int N = (c->unit_kind == 0) ? c->H * c->dk : c->H;
    size_t base = (size_t)b * N;
    int gsz = c->group_heads * c->dk;
    int kind = c->weight_kind;
    if (kind < 0 || kind > 8) return ORC_EINVAL;
    int A = 0, B0 = 0;
    orc_shuffle(N, &A, &B0);
    float mean = 0.0f;
    for (int u = 0; u < N; u++) {
        if (c->unit_kind == 0 && u % gsz == 0) {   /* mean R^2 of the group starting here */
            float acc = 0.0f;
            for (int r = u; r < u + gsz; r++) acc = acc + range[base + r] * range[base + r];
            mean = acc / (float)gsz;
        }
        float R2 = 1.0f, rt2 = 1.0f;
        if (c->unit_kind == 0) {
            R2 = range[base + u] * range[base + u];
            if (mean > 0.0f) rt2 = R2 / mean;
        }
        int us = (kind == 7) ? (int)(((long long)A * u + B0) % N) : u;
        float w = weight_of(c, kind, ema_s[base + us], ema_r[base + us], R2, rt2);
        if (w > 0x1p60f) w = 0x1p60f;
        cw[u] = (w >= 0x1p-60f) ? w : -1.0f;  /* -1 flags the null weight 2^-200 (also NaN) */
    }
    return ORC_OK;
}

/* Exact marginal value of the b-th bit of unit u: c_u 4^{-b}, as a double (exact: c is an
 * FP32 number, the scaling a power of two).  The null weight is 2^-200. */
static double bit_value(const float* cw, int u, int b) {
    double cv = (cw[u] < 0.0f) ? 0x1p-200 : (double)cw[u];
    return ldexp(cv, -2 * b);
}

/* Total order on bits: higher value first; equal value -> lower unit index first; within a
 * unit, lower bit first (values strictly decrease with b, except for the null weight whose
 * bits are ordered by b then by unit).  Returns 1 if bit (u1, b1) ranks above (u2, b2). */
static int ranks_above(const float* cw, int u1, int b1, int u2, int b2) {
    double v1 = bit_value(cw, u1, b1), v2 = bit_value(cw, u2, b2);
    if (v1 != v2) return v1 > v2;
    if (u1 != u2) return u1 < u2;
    return b1 < b2;
}

/* Eq. (4) and the integer rounding that follows it: "round, clip to [b_min, b_max], and
 * adjust widths to meet the layer budget".
 *   1. real-valued widths b_i = bbar + 1/2 log2(c_i / GM(c)) (FP64; null weights start at
 *      b_min and are left out of GM);
 *   2. round to nearest; 3. clip;
 *   4. adjust to the budget: while over it, take back the lowest-ranked bit held; while
 *      under it, grant the highest-ranked bit not yet held;
 *   5. while the lowest-ranked held bit ranks below the highest-ranked free bit, move it
 *      (the adjustment ends at the minimum of the high-rate proxy sum c_i 4^{-b_i}).
 * The result is the top-M bits of the order above, M = budget - N b_min. */
int orc_alloc_from_weights(int N, const float* cw, int bmin, int bmax, long total, int bbar_num,
                           int bbar_den, uint8_t* widths) {
    if ((long)N * bmin > total || (long)N * bmax < total) return ORC_EBUDGET;
    int* bw = (int*)malloc(sizeof(int) * N);
    double bbar = (double)bbar_num / (double)bbar_den, lsum = 0.0;
    int npos = 0;
    for (int u = 0; u < N; u++)
        if (cw[u] > 0.0f) {
            lsum += log2((double)cw[u]);
            npos++;
        }
    double lgm = npos ? lsum / npos : 0.0;
    long sum = 0;
    for (int u = 0; u < N; u++) {
        int b = bmin;
        if (cw[u] > 0.0f) {
            double br = bbar + 0.5 * (log2((double)cw[u]) - lgm);
            double r = floor(br + 0.5);
            if (r < bmin) r = bmin;
            if (r > bmax) r = bmax;
            b = (int)r;
        }
        bw[u] = b;
        sum += b;
    }
    while (sum > total) {          /* take back the lowest-ranked held bit */
        int lo = -1;
        for (int u = 0; u < N; u++)
            if (bw[u] > bmin && (lo < 0 || ranks_above(cw, lo, bw[lo], u, bw[u]))) lo = u;
        bw[lo]--;
        sum--;
    }
    while (sum < total) {          /* grant the highest-ranked free bit */
        int hi = -1;
        for (int u = 0; u < N; u++)
            if (bw[u] < bmax && (hi < 0 || ranks_above(cw, u, bw[u] + 1, hi, bw[hi] + 1))) hi = u;
        bw[hi]++;
        sum++;
    }
    for (;;) {                     /* exchange until no held bit ranks below a free bit */
        int lo = -1, hi = -1;
        for (int u = 0; u < N; u++) {
            if (bw[u] > bmin && (lo < 0 || ranks_above(cw, lo, bw[lo], u, bw[u]))) lo = u;
            if (bw[u] < bmax && (hi < 0 || ranks_above(cw, u, bw[u] + 1, hi, bw[hi] + 1))) hi = u;
        }
        if (lo < 0 || hi < 0 || lo == hi) break;
        if (!ranks_above(cw, hi, bw[hi] + 1, lo, bw[lo])) break;
        bw[lo]--;
        bw[hi]++;
    }
    for (int u = 0; u < N; u++) widths[u] = (uint8_t)bw[u];
    free(bw);
    return ORC_OK;
}

/* Allocation for every batch element: weights (Eq. 3) -> widths (Eq. 4 + rounding) ->
 * head offsets (prefix sums of row bytes).  Budget: sum of widths = N bbar per element. */
int orc_alloc(const orc_cfg* c, const float* ema_s, const float* ema_r, const float* range,
              uint8_t* widths, uint32_t* head_off) {
    int N = (c->unit_kind == 0) ? c->H * c->dk : c->H;
    long num = (long)N * c->bbar_num;
    if (num % c->bbar_den) return ORC_EINVAL;
    long total = num / c->bbar_den;
    float* cw = (float*)malloc(sizeof(float) * N);
    for (int b = 0; b < c->B; b++) {
        int rcw = orc_weights(c, b, ema_s, ema_r, range, cw);
        if (rcw) {
            free(cw);
            return rcw;
        }
        int rc = orc_alloc_from_weights(N, cw, c->bmin, c->bmax, total, c->bbar_num, c->bbar_den,
                                        widths + (size_t)b * N);
        if (rc) {
            free(cw);
            return rc;
        }
        uint32_t off = 0;
        for (int h = 0; h < c->H; h++) {
            head_off[(size_t)b * c->H + h] = off;
            for (int i = 0; i < c->dk; i++) off += (uint32_t)(unit_width(c, widths, b, h, i) * c->dv / 8);
        }
    }
    free(cw);
    return ORC_OK;
}

/* Initial widths: the allocation with every weight equal (uniform bbar when it is an
 * integer), offsets to match. */
int orc_init_widths(const orc_cfg* c, uint8_t* widths, uint32_t* head_off) {
    int N = (c->unit_kind == 0) ? c->H * c->dk : c->H;
    long num = (long)N * c->bbar_num;
    if (num % c->bbar_den) return ORC_EINVAL;
    float* cw = (float*)malloc(sizeof(float) * N);
    for (int u = 0; u < N; u++) cw[u] = 1.0f;
    for (int b = 0; b < c->B; b++) {
        int rc = orc_alloc_from_weights(N, cw, c->bmin, c->bmax, num / c->bbar_den, c->bbar_num,
                                        c->bbar_den, widths + (size_t)b * N);
        if (rc) {
            free(cw);
            return rc;
        }
        uint32_t off = 0;
        for (int h = 0; h < c->H; h++) {
            head_off[(size_t)b * c->H + h] = off;
            for (int i = 0; i < c->dk; i++) off += (uint32_t)(unit_width(c, widths, b, h, i) * c->dv / 8);
        }
    }
    free(cw);
    return ORC_OK;
}

/* ---------------------------------------------------------------------------------------
 * Sec. 3, "Decay-gate quantization": levels uniform in log s per channel.
 * For channel ch (over `count` samples s[n * nchan + ch], all > 0): lo = log min s,
 * hi = log max s, L = 2^g levels l_k = exp(lo + k (hi - lo) / (L - 1)) (l_0 = min s and
 * l_{L-1} = max s exactly), thresholds theta_k = exp(lo + (k - 1/2)(hi - lo)/(L - 1)) for
 * k = 1..L-1 (geometric means of neighbouring levels).  Levels and thresholds are computed
 * in FP64 and rounded to FP32; code = #{k : s >= theta_k} in FP32; ties go up.
 * ------------------------------------------------------------------------------------- */
int orc_quant_decay(long count, int nchan, const float* s, int g, uint8_t* codes, float* lut,
                    float* thr) {
    if (g < 1 || g > 8) return ORC_EINVAL;
    int L = 1 << g;
    float* th = (float*)malloc(sizeof(float) * (L > 1 ? L - 1 : 1));
    for (int ch = 0; ch < nchan; ch++) {
        float mn = INFINITY, mx = 0.0f;
        for (long n = 0; n < count; n++) {
            float x = s[(size_t)n * nchan + ch];
            if (!(x > 0.0f) || !isfinite(x)) {
                free(th);
                return ORC_EINVAL;
            }
            if (x < mn) mn = x;
            if (x > mx) mx = x;
        }
        double lo = log((double)mn), hi = log((double)mx), step = (hi - lo) / (double)(L - 1);
        for (int k = 0; k < L; k++) lut[(size_t)ch * L + k] = (float)exp(lo + k * step);
        lut[(size_t)ch * L] = mn;
        lut[(size_t)ch * L + L - 1] = mx;
        for (int k = 1; k < L; k++) {
            th[k - 1] = (float)exp(lo + ((double)k - 0.5) * step);
            if (thr) thr[(size_t)ch * (L - 1) + k - 1] = th[k - 1];
        }
        for (long n = 0; n < count; n++) {
            float x = s[(size_t)n * nchan + ch];
            int code = 0;
            for (int k = 1; k < L; k++)
                if (x >= th[k - 1]) code++;
            codes[(size_t)n * nchan + ch] = (uint8_t)code;
        }
    }
    free(th);
    return ORC_OK;
}

/* ---------------------------------------------------------------------------------------
 * One write-back interval (Sec. 2, "Accumulated readout error", and the protocol of Sec. 5):
 * for every head, unpack + dequantise the state written at the previous write-back, run the
 * tokens t_begin..t_end-1 of Eq. (1) in FP32 (readouts o_t are taken before quantising),
 * update the EMA statistics (Sec. 3), then requantise + repack with the target widths.
 *
 * Inputs are the full (B, T, H, .) tensors; s is (B, T, H, dk) for per-row rates and
 * (B, T, H) for per-head rates; with s_code/s_lut the rate is s_lut[ch * 2^g + code].
 * EMA per token (span 64): alpha = 2 / (span + 1), m <- m + alpha (x - m), the first token
 * of the sequence (t = 0) initialising m = x; x_s = 1 - e^{-2 s}, x_r = beta (2 - beta) k_i^2
 * (row unit) or beta (2 - beta) |k|^2 / dk (head unit), 0 without erasure.  With general
 * erasure (erase_kind 2) a_tok (B, T, H, dk) and w_tok (B, T, H, dv) give a and w per token
 * and x_r = 2 a_i k_i - a_i^2 |k|^2 (row unit) or its mean over the rows (head unit): the
 * fraction of row i's error energy that (I - k a^T) removes, beta (2 - beta) k_i^2 for
 * a = beta k and |k| = 1.
 * The range factor is refitted when fit_every <= 1 or (w_index + h) % fit_every == 0, else
 * the factor stored at the previous write-back (fidx_in) is reused.
 * x_dump (optional) receives the FP32 state before quantisation (B, H, dk, dv).
 * ------------------------------------------------------------------------------------- */
int orc_step(const orc_cfg* c, const uint8_t* pay_in, const uint16_t* sc_in, const uint8_t* w_in,
             const uint32_t* off_in, const uint8_t* fidx_in, uint8_t* pay_out, uint16_t* sc_out,
             const uint8_t* w_out, const uint32_t* off_out, uint8_t* fidx_out, int T, int t_begin,
             int t_end, int w_index, const float* q, const float* k, const float* v,
             const float* s, const uint8_t* s_code, const float* s_lut, const float* beta,
             float* o, float* ema_s, float* ema_r, float* range, float* x_dump,
             const float* a_tok, const float* w_tok) {
    int H = c->H, dk = c->dk, dv = c->dv, L = 1 << c->gate_bits;
    long rb = orc_region_bytes(c);
    if (rb < 0 || !layout_ok(c, w_in, off_in) || !layout_ok(c, w_out, off_out)) return ORC_EINVAL;
    if (c->erase_kind == 2 && (!a_tok || !w_tok)) return ORC_EINVAL;
    float alpha = 2.0f / (c->ema_span + 1.0f);
    memset(pay_out, 0, (size_t)c->B * (size_t)rb);
    /* Heads are independent within a write-back (each writes only its own bytes, scales,
     * statistics and readouts), so the timing build (ORC_OPENMP) shares them out over threads;
     * every head's arithmetic is the same sequential code either way. */
    const int nbh = c->B * H;
#ifdef ORC_OPENMP
#pragma omp parallel
#endif
    {
    float* X = (float*)malloc(sizeof(float) * (size_t)dk * dv);
    float* d = (float*)malloc(sizeof(float) * dk);
    float* p = (float*)malloc(sizeof(float) * dv);
#ifdef ORC_OPENMP
#pragma omp for schedule(dynamic, 1)
#endif
    for (int bh = 0; bh < nbh; bh++) {
        const int b = bh / H, h = bh % H;
        {
            unpack_head(c, b, h, pay_in, sc_in, w_in, off_in, X);
            for (int t = t_begin; t < t_end; t++) {
                size_t tok = ((size_t)b * T + t) * H + h;
                const float *kt = k + tok * dk, *qt = q + tok * dk, *vt = v + tok * dv;
                float bt = (c->erase_kind == 0) ? beta[tok] : 1.0f;
                /* general erasure (erase_kind 2): a, w given; its statistic per row is
                 * 2 a_i k_i - a_i^2 |k|^2 (|k|^2 summed in index order) */
                const float *at = (c->erase_kind == 2) ? a_tok + tok * dk : 0;
                const float *wt = (c->erase_kind == 2) ? w_tok + tok * dv : 0;
                float ksq = 0.0f;
                for (int i = 0; i < dk; i++) ksq = ksq + kt[i] * kt[i];
                float ssum = 0.0f;
                for (int i = 0; i < dk; i++) {
                    int ch = (c->decay_kind == 0) ? h * dk + i : h;
                    size_t si = (c->decay_kind == 0) ? tok * dk + i : tok;
                    float si_rate = s_code ? s_lut[(size_t)ch * L + s_code[si]] : s[si];
                    d[i] = expf(-si_rate);
                    /* EMA statistics, row unit */
                    if (c->unit_kind == 0) {
                        size_t u = ((size_t)b * H + h) * dk + i;
                        float xs = -expm1f(-2.0f * si_rate);
                        float xr = (c->erase_kind == 0) ? (bt * (2.0f - bt)) * (kt[i] * kt[i]) : 0.0f;
                        if (c->erase_kind == 2) xr = 2.0f * (at[i] * kt[i]) - (at[i] * at[i]) * ksq;
                        if (t == 0) {
                            ema_s[u] = xs;
                            ema_r[u] = xr;
                        } else {
                            ema_s[u] = ema_s[u] + alpha * (xs - ema_s[u]);
                            ema_r[u] = ema_r[u] + alpha * (xr - ema_r[u]);
                        }
                    }
                    ssum = ssum + kt[i] * kt[i];
                }
                if (c->unit_kind == 1) {
                    size_t u = (size_t)b * H + h;
                    float xs = -expm1f(-2.0f * (s_code ? s_lut[(size_t)h * L + s_code[tok]] : s[tok]));
                    float xr = (c->erase_kind == 0) ? (bt * (2.0f - bt)) * (ssum / (float)dk) : 0.0f;
                    if (c->erase_kind == 2) {   /* mean over rows of 2 a_i k_i - a_i^2 |k|^2 */
                        float ak = 0.0f, aa = 0.0f;
                        for (int i = 0; i < dk; i++) {
                            ak = ak + at[i] * kt[i];
                            aa = aa + at[i] * at[i];
                        }
                        xr = (2.0f * ak - aa * ksq) / (float)dk;
                    }
                    if (t == 0) {
                        ema_s[u] = xs;
                        ema_r[u] = xr;
                    } else {
                        ema_s[u] = ema_s[u] + alpha * (xs - ema_s[u]);
                        ema_r[u] = ema_r[u] + alpha * (xr - ema_r[u]);
                    }
                }
                /* Eq. (1): S' = D S; KDA / GDN: a = beta k, w = beta 1; Mamba-2: a = 0, w = 1 */
                for (int i = 0; i < dk; i++)
                    for (int j = 0; j < dv; j++) X[(size_t)i * dv + j] = X[(size_t)i * dv + j] * d[i];
                if (c->erase_kind == 0) {
                    for (int j = 0; j < dv; j++) {
                        float acc = 0.0f;
                        for (int i = 0; i < dk; i++) acc = acc + (bt * kt[i]) * X[(size_t)i * dv + j];
                        p[j] = acc;
                    }
                    for (int i = 0; i < dk; i++)
                        for (int j = 0; j < dv; j++)
                            X[(size_t)i * dv + j] =
                                (X[(size_t)i * dv + j] - kt[i] * p[j]) + kt[i] * (bt * vt[j]);
                } else if (c->erase_kind == 2) {   /* Eq. (1) with the given a and w */
                    for (int j = 0; j < dv; j++) {
                        float acc = 0.0f;
                        for (int i = 0; i < dk; i++) acc = acc + at[i] * X[(size_t)i * dv + j];
                        p[j] = acc;
                    }
                    for (int i = 0; i < dk; i++)
                        for (int j = 0; j < dv; j++)
                            X[(size_t)i * dv + j] =
                                (X[(size_t)i * dv + j] - kt[i] * p[j]) + kt[i] * (wt[j] * vt[j]);
                } else {
                    for (int i = 0; i < dk; i++)
                        for (int j = 0; j < dv; j++)
                            X[(size_t)i * dv + j] = X[(size_t)i * dv + j] + kt[i] * vt[j];
                }
                for (int j = 0; j < dv; j++) {   /* outputs precede quantisation */
                    float acc = 0.0f;
                    for (int i = 0; i < dk; i++) acc = acc + X[(size_t)i * dv + j] * qt[i];
                    o[tok * dv + j] = acc;
                }
            }
            if (x_dump) memcpy(x_dump + ((size_t)b * H + h) * dk * dv, X, sizeof(float) * dk * dv);
            int refit = (c->fit_every <= 1) || ((w_index + h) % c->fit_every == 0);
            pack_head(c, b, h, X, w_out, off_out, refit, fidx_in, pay_out, sc_out, fidx_out, range);
        }
    }
    free(X);
    free(d);
    free(p);
    }
    return ORC_OK;
}

/* ---------------------------------------------------------------------------------------
 * One write-back with the allocation taken from this write-back's own statistics (the
 * reading of Eq. 3 that uses the ranges of the state being quantised; Sec. 3):
 *   1. run the interval's tokens for every head (orc_step into scratch buffers laid out like
 *      the input), which updates the EMAs and ranges and writes the readouts;
 *   2. allocate widths and head offsets from those statistics (orc_alloc) into w_out/off_out;
 *   3. quantise + pack every head's state with the new widths.
 * ------------------------------------------------------------------------------------- */
int orc_step_current(const orc_cfg* c, const uint8_t* pay_in, const uint16_t* sc_in,
                     const uint8_t* w_in, const uint32_t* off_in, const uint8_t* fidx_in,
                     uint8_t* pay_out, uint16_t* sc_out, uint8_t* w_out, uint32_t* off_out,
                     uint8_t* fidx_out, int T, int t_begin, int t_end, int w_index,
                     const float* q, const float* k, const float* v, const float* s,
                     const uint8_t* s_code, const float* s_lut, const float* beta, float* o,
                     float* ema_s, float* ema_r, float* range, float* x_dump,
                     const float* a_tok, const float* w_tok) {
    if (c->unit_kind != 0) return ORC_EINVAL;
    int H = c->H, dk = c->dk, dv = c->dv;
    long rb = orc_region_bytes(c);
    if (rb < 0) return ORC_EINVAL;
    size_t n_el = (size_t)c->B * H * dk * dv, n_sc = (size_t)c->B * H * dk;
    float* X = (float*)malloc(sizeof(float) * n_el);
    uint8_t* pay_tmp = (uint8_t*)malloc((size_t)c->B * rb);
    uint16_t* sc_tmp = (uint16_t*)malloc(sizeof(uint16_t) * n_sc);
    uint8_t* fidx_tmp = (uint8_t*)malloc(n_sc);
    int rc = orc_step(c, pay_in, sc_in, w_in, off_in, fidx_in, pay_tmp, sc_tmp, w_in, off_in,
                      fidx_tmp, T, t_begin, t_end, w_index, q, k, v, s, s_code, s_lut, beta, o,
                      ema_s, ema_r, range, X, a_tok, w_tok);
    if (rc == ORC_OK) rc = orc_alloc(c, ema_s, ema_r, range, w_out, off_out);
    if (rc == ORC_OK && !layout_ok(c, w_out, off_out)) rc = ORC_EINVAL;
    if (rc == ORC_OK) {
        memset(pay_out, 0, (size_t)c->B * rb);
        for (int b = 0; b < c->B; b++)
            for (int h = 0; h < H; h++) {
                int refit = (c->fit_every <= 1) || ((w_index + h) % c->fit_every == 0);
                pack_head(c, b, h, X + ((size_t)b * H + h) * dk * dv, w_out, off_out, refit,
                          fidx_in, pay_out, sc_out, fidx_out, range);
            }
        if (x_dump) memcpy(x_dump, X, sizeof(float) * n_el);
    }
    free(X);
    free(pay_tmp);
    free(sc_tmp);
    free(fidx_tmp);
    return rc;
}
