/*
 * Log_bQuant reference oracle -- TEST INFRASTRUCTURE ONLY.
 *
 * A plain, slow, obviously correct CPU restatement of what the Log_bQuant
 * inference path computes, written in fp64 from the paper's definitions:
 *
 *   Eq. (1)  Quant(b, s, x)   = 0 if x = 0, else sign(x) * round_clamp(log_b|x| + s)
 *   Eq. (2)  Dequant(b, s, q) = 0 if q = 0, else sign(q) * b^(|q| - s)
 *   Sec. 3.1 q_max = 2^(n-1) - 1, one codebook (b, s) per weight matrix
 *   Eq. (3)  b = (w_max / w_min)^(1 / q_max)
 *   Eq. (4)  s = q_max - floor(log_b w_max)
 *   Eq. (5)  w_min = min{ t : sum_{|w_i| <= t} w_i^2 / sum_i w_i^2 >= eps }
 *   Sec. 3.3 dequantisation through a lookup table; packed low-bit weights
 *
 * Only the test suite, the smoke check and the CPU-baseline leg of the
 * benchmark may load this file.  It shares no code, header, table or
 * constant generator with the CUDA library; both sides are written
 * independently from the same definitions and from the packed-code layout
 * spelled out below.
 *
 * Readings of points the paper leaves open (each one is a choice):
 *   R1  The clamp of Eq. (1) acts on the magnitude: m = clamp(round(t), 0, q_max).
 *       A weight below the lowest decision boundary maps to code 0 (pruned).
 *   R2  Rounding ties go up in magnitude (t = j + 1/2 -> j + 1).
 *   R3  Rounding happens in log space (Eq. (1) rounds log_b|x|), so decision
 *       boundaries are geometric midpoints tau_j = b^(j + 1/2 - s).
 *   R4  Shift mode EXACT (default): s = q_max - log_b(range), so the top level
 *       equals the range.  Shift mode FLOOR: Eq. (4) literally,
 *       s = q_max - floor(log_b range), floor taken as the largest integer e
 *       with b^e <= range.
 *   R5  The dequantised value used by a linear layer is the fp32 level
 *       rounded (nearest-even) to the activation dtype (bf16 or fp16); the
 *       fp32 level itself is the fp64 level rounded to nearest-even.
 *
 * Packed code layout (the library must produce exactly these bytes):
 *   code of a weight = sign << (n-1) | m, sign = 1 for negative weights with
 *   m > 0 (the code 1 << (n-1), "-0", is never produced).
 *   n = 4: row-major [N][K/2] bytes; byte j of a row holds k = 2j in its low
 *          nibble and k = 2j+1 in its high nibble.
 *   n = 3: row-major [N][3K/8] bytes; every 32 consecutive k form a 12-byte
 *          group of three little-endian uint32 words W0, W1, W2.  Pair p
 *          (k = 2p, 2p+1 within the group) has the 6-bit field
 *          f_p = code(2p) | code(2p+1) << 3.  For p = 5i + j (i < 3, j < 5)
 *          f_p sits in bits [6j, 6j+6) of W_i; f_15 is split two bits per
 *          word: bits 30-31 of W0, W1, W2 hold f_15 bits 0-1, 2-3, 4-5.
 *   n = 8: row-major [N][K] bytes, one code per byte (sign in bit 7).
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

#define ORACLE_SHIFT_EXACT 0
#define ORACLE_SHIFT_FLOOR 1

typedef struct {
    int32_t bits;          /* n */
    int32_t qmax;          /* q_max = 2^(n-1) - 1 */
    int32_t shift_mode;    /* ORACLE_SHIFT_EXACT or ORACLE_SHIFT_FLOOR */
    int32_t _pad;
    double base;           /* b */
    double range;          /* w_max handed in */
    double shift;          /* s */
    double level[128];     /* L_m = b^(m - s), m = 0..q_max, L_0 = 0 (Eq. (2)) */
    double tau[128];       /* tau_j = b^(j + 1/2 - s), j = 0..q_max-1 (R3) */
    float level32[128];    /* L_m rounded to nearest-even fp32 */
    float tau32_up[128];   /* smallest fp32 >= tau_j */
    uint16_t level_bf16[128];/* level32 rounded to nearest-even bf16 (bits) */
    uint16_t level_f16[128]; /* level32 rounded to nearest-even fp16 (bits) */
} oracle_codebook;

/* ------------------------------------------------------------------ */
/* Rounding of a real value to a binary floating-point format, written  */
/* from the IEEE-754 definition: p significand bits (implicit one       */
/* included), smallest normal exponent emin (value 2^emin), largest     */
/* finite value, subnormals with quantum 2^(emin - p + 1).  Ties go to  */
/* the even significand.  Returns the rounded real value.               */
/* ------------------------------------------------------------------ */
static double round_to_format(double v, int p, int emin, double maxfinite)
{
    if (v == 0.0 || isnan(v) || isinf(v)) return v;
    double a = fabs(v);
    int e;
    frexp(a, &e);                 /* a = f * 2^e, f in [0.5, 1) -> a in [2^(e-1), 2^e) */
    int exp_unbiased = e - 1;     /* a in [2^exp_unbiased, 2^(exp_unbiased+1)) */
    if (exp_unbiased < emin) exp_unbiased = emin;   /* subnormal range: fixed quantum */
    double quantum = ldexp(1.0, exp_unbiased - (p - 1));
    double scaled = a / quantum;  /* exact: division by a power of two */
    double fl = floor(scaled);
    double frac = scaled - fl;
    double r;
    if (frac > 0.5) r = fl + 1.0;
    else if (frac < 0.5) r = fl;
    else r = (fmod(fl, 2.0) == 0.0) ? fl : fl + 1.0;
    double out = r * quantum;
    if (out > maxfinite) out = INFINITY;
    return v < 0 ? -out : out;
}

double oracle_round_f32(double v)  { return round_to_format(v, 24, -126, 3.4028234663852886e38); }
double oracle_round_bf16(double v) { return round_to_format(v, 8, -126, 3.3895313892515355e38); }
double oracle_round_f16(double v)  { return round_to_format(v, 11, -14, 65504.0); }

/* Encode a value that is already representable in a 16-bit format with
 * exponent width ebits and mantissa width mbits into its bit pattern. */
static uint16_t encode16(double v, int ebits, int mbits)
{
    uint16_t sign = (signbit(v) ? 1u : 0u) << 15;
    double a = fabs(v);
    int bias = (1 << (ebits - 1)) - 1;
    if (a == 0.0) return sign;
    if (isinf(a)) return sign | (uint16_t)(((1u << ebits) - 1u) << mbits);
    int e;
    frexp(a, &e);
    int E = e - 1;                         /* a = 1.f * 2^E */
    int emin = 1 - bias;
    if (E < emin) {                        /* subnormal: a = frac * 2^(emin - mbits) */
        double mant = a / ldexp(1.0, emin - mbits);
        return sign | (uint16_t)mant;
    }
    double mant = (a / ldexp(1.0, E) - 1.0) * ldexp(1.0, mbits);
    return sign | (uint16_t)((uint32_t)(E + bias) << mbits) | (uint16_t)mant;
}

uint16_t oracle_bf16_bits(double v) { return encode16(oracle_round_bf16(v), 8, 7); }
uint16_t oracle_f16_bits(double v)  { return encode16(oracle_round_f16(v), 5, 10); }

/* Smallest fp32 value >= t (t > 0), found by stepping the nearest fp32. */
static float f32_round_up(double t)
{
    float f = (float)oracle_round_f32(t);
    while ((double)f < t) f = nextafterf(f, INFINITY);
    while (1) {
        float g = nextafterf(f, 0.0f);
        if ((double)g >= t) f = g; else break;
    }
    return f;
}

/* Largest integer e with b^e <= x (x > 0, b > 1): the floor of log_b x,
 * settled by comparing powers so that exact powers of b land correctly. */
static long floor_log_b(double x, double b)
{
    long e = (long)floor(log(x) / log(b));
    while (pow(b, (double)(e + 1)) <= x) e++;
    while (pow(b, (double)e) > x) e--;
    return e;
}

/* Codebook of Sec. 3.1: levels from Eq. (2), shift from Eq. (4) (R4). */
int oracle_build_codebook(int bits, double base, double range, int shift_mode,
                          oracle_codebook* cb)
{
    if ((bits != 3 && bits != 4 && bits != 8) || !(base > 1.0) || !isfinite(base) ||
        !(range > 0.0) || !isfinite(range))
        return 1;
    memset(cb, 0, sizeof *cb);
    cb->bits = bits;
    cb->qmax = (1 << (bits - 1)) - 1;
    cb->shift_mode = shift_mode;
    cb->base = base;
    cb->range = range;
    double lb_range = log(range) / log(base);
    if (shift_mode == ORACLE_SHIFT_FLOOR)
        cb->shift = (double)cb->qmax - (double)floor_log_b(range, base);
    else
        cb->shift = (double)cb->qmax - lb_range;
    for (int m = 0; m <= cb->qmax; ++m) {
        /* b^(m - s).  In exact mode m - s = m - q_max + log_b(range), written
         * as range * b^(m - q_max) so the top level is the range itself. */
        double L;
        if (m == 0) L = 0.0;
        else if (shift_mode == ORACLE_SHIFT_FLOOR)
            L = pow(base, (double)m - cb->shift);
        else
            L = range * pow(base, (double)(m - cb->qmax));
        cb->level[m] = L;
        cb->level32[m] = (float)oracle_round_f32(L);
        cb->level_bf16[m] = oracle_bf16_bits((double)cb->level32[m]);
        cb->level_f16[m] = oracle_f16_bits((double)cb->level32[m]);
    }
    for (int j = 0; j < cb->qmax; ++j) {
        double t;
        if (shift_mode == ORACLE_SHIFT_FLOOR)
            t = pow(base, (double)j + 0.5 - cb->shift);
        else
            t = range * pow(base, (double)j + 0.5 - (double)cb->qmax);
        cb->tau[j] = t;
        cb->tau32_up[j] = f32_round_up(t);
    }
    return 0;
}

/* Route 1 -- Eq. (1) as printed: t = log_b|x| + s, rounded (R2), clamped (R1). */
void oracle_quantize_log(const float* w, int64_t n, const oracle_codebook* cb, int8_t* q)
{
    double lnb = log(cb->base);
    for (int64_t i = 0; i < n; ++i) {
        double x = (double)w[i];
        if (x == 0.0) { q[i] = 0; continue; }
        double t = log(fabs(x)) / lnb + cb->shift;
        double r = floor(t + 0.5);
        if (r < 0.0) r = 0.0;
        if (r > (double)cb->qmax) r = (double)cb->qmax;
        int m = (int)r;
        q[i] = (int8_t)(x < 0 ? -m : m);
    }
}

/* Route 2 -- brute force: the level index j in 0..q_max nearest to
 * t = log_b|x| + s (ties to the larger j), i.e. argmin over all levels. */
void oracle_quantize_argmin(const float* w, int64_t n, const oracle_codebook* cb, int8_t* q)
{
    double lnb = log(cb->base);
    for (int64_t i = 0; i < n; ++i) {
        double x = (double)w[i];
        if (x == 0.0) { q[i] = 0; continue; }
        double t = log(fabs(x)) / lnb + cb->shift;
        int best = 0;
        double bestd = fabs(t - 0.0);
        for (int j = 1; j <= cb->qmax; ++j) {
            double d = fabs(t - (double)j);
            if (d <= bestd) { bestd = d; best = j; }
        }
        q[i] = (int8_t)(x < 0 ? -best : best);
    }
}

/* Route 3 -- decision boundaries: m = #{ j : |x| >= tau_j } with the fp64
 * boundaries of R3 (no logarithm of the weight is taken). */
void oracle_quantize_thresh(const float* w, int64_t n, const oracle_codebook* cb, int8_t* q)
{
    for (int64_t i = 0; i < n; ++i) {
        double a = fabs((double)w[i]);
        int m = 0;
        for (int j = 0; j < cb->qmax; ++j)
            if (a >= cb->tau[j]) m++;
        q[i] = (int8_t)(w[i] < 0 ? -m : m);
    }
}

/* max_i |w_i| (Sec. 3.2, w_max) and a flag for NaN / Inf entries. */
double oracle_absmax(const float* w, int64_t n, int* nonfinite)
{
    double mx = 0.0;
    int bad = 0;
    for (int64_t i = 0; i < n; ++i) {
        double a = fabs((double)w[i]);
        if (!isfinite(a)) { bad = 1; continue; }
        if (a > mx) mx = a;
    }
    if (nonfinite) *nonfinite = bad;
    return mx;
}

static unsigned code_of(int8_t qv, int bits)
{
    unsigned m = (unsigned)(qv < 0 ? -qv : qv);
    unsigned s = (qv < 0) ? 1u : 0u;
    return (s << (bits - 1)) | m;
}

static int8_t value_of(unsigned code, int bits)
{
    unsigned m = code & ((1u << (bits - 1)) - 1u);
    unsigned s = (code >> (bits - 1)) & 1u;
    return (int8_t)(s ? -(int)m : (int)m);
}

int64_t oracle_packed_row_bytes(int64_t K, int bits)
{
    if (bits == 8) return K;
    if (bits == 4) return K / 2;
    if (bits == 3) return (K / 32) * 12;
    return -1;
}

/* Pack signed integer codes q[N][K] into the layout described above. */
int oracle_pack(const int8_t* q, int64_t N, int64_t K, int bits, uint8_t* out)
{
    int64_t rb = oracle_packed_row_bytes(K, bits);
    if (rb < 0) return 1;
    for (int64_t r = 0; r < N; ++r) {
        const int8_t* qr = q + r * K;
        uint8_t* o = out + r * rb;
        if (bits == 8) {
            for (int64_t k = 0; k < K; ++k) o[k] = (uint8_t)code_of(qr[k], 8);
        } else if (bits == 4) {
            for (int64_t j = 0; j < K / 2; ++j)
                o[j] = (uint8_t)(code_of(qr[2 * j], 4) | (code_of(qr[2 * j + 1], 4) << 4));
        } else {
            if (K % 32) return 1;
            for (int64_t g = 0; g < K / 32; ++g) {
                uint32_t W[3] = {0, 0, 0};
                for (int p = 0; p < 16; ++p) {
                    uint32_t f = code_of(qr[32 * g + 2 * p], 3) |
                                 (code_of(qr[32 * g + 2 * p + 1], 3) << 3);
                    if (p < 15) {
                        W[p / 5] |= f << (6 * (p % 5));
                    } else {
                        W[0] |= (f & 3u) << 30;
                        W[1] |= ((f >> 2) & 3u) << 30;
                        W[2] |= ((f >> 4) & 3u) << 30;
                    }
                }
                for (int i = 0; i < 3; ++i)
                    for (int b = 0; b < 4; ++b)
                        o[12 * g + 4 * i + b] = (uint8_t)(W[i] >> (8 * b));
            }
        }
    }
    return 0;
}

/* Inverse of oracle_pack. */
int oracle_unpack(const uint8_t* packed, int64_t N, int64_t K, int bits, int8_t* q)
{
    int64_t rb = oracle_packed_row_bytes(K, bits);
    if (rb < 0) return 1;
    for (int64_t r = 0; r < N; ++r) {
        const uint8_t* p = packed + r * rb;
        int8_t* qr = q + r * K;
        if (bits == 8) {
            for (int64_t k = 0; k < K; ++k) qr[k] = value_of(p[k], 8);
        } else if (bits == 4) {
            for (int64_t j = 0; j < K / 2; ++j) {
                qr[2 * j] = value_of(p[j] & 0xFu, 4);
                qr[2 * j + 1] = value_of(p[j] >> 4, 4);
            }
        } else {
            for (int64_t g = 0; g < K / 32; ++g) {
                uint32_t W[3];
                for (int i = 0; i < 3; ++i)
                    W[i] = (uint32_t)p[12 * g + 4 * i] | ((uint32_t)p[12 * g + 4 * i + 1] << 8) |
                           ((uint32_t)p[12 * g + 4 * i + 2] << 16) | ((uint32_t)p[12 * g + 4 * i + 3] << 24);
                for (int pi = 0; pi < 16; ++pi) {
                    uint32_t f;
                    if (pi < 15) f = (W[pi / 5] >> (6 * (pi % 5))) & 0x3Fu;
                    else f = (W[0] >> 30) | ((W[1] >> 30) << 2) | ((W[2] >> 30) << 4);
                    qr[32 * g + 2 * pi] = value_of(f & 7u, 3);
                    qr[32 * g + 2 * pi + 1] = value_of(f >> 3, 3);
                }
            }
        }
    }
    return 0;
}

/* Eq. (2) through the lookup table of Sec. 3.3.  table selects which copy
 * of the levels is read: 0 = fp64 levels, 1 = fp32, 2 = bf16, 3 = fp16. */
static double bits16_value(uint16_t h, int ebits, int mbits)
{
    int bias = (1 << (ebits - 1)) - 1;
    int s = h >> 15;
    int E = (h >> mbits) & ((1 << ebits) - 1);
    int M = h & ((1 << mbits) - 1);
    double v;
    if (E == 0) v = ldexp((double)M, 1 - bias - mbits);
    else v = ldexp(1.0 + ldexp((double)M, -mbits), E - bias);
    return s ? -v : v;
}

void oracle_dequant(const int8_t* q, int64_t n, const oracle_codebook* cb, int table, double* out)
{
    for (int64_t i = 0; i < n; ++i) {
        int m = q[i] < 0 ? -q[i] : q[i];
        double mag;
        switch (table) {
        case 1: mag = (double)cb->level32[m]; break;
        case 2: mag = bits16_value(cb->level_bf16[m], 8, 7); break;
        case 3: mag = bits16_value(cb->level_f16[m], 5, 10); break;
        default: mag = cb->level[m]; break;
        }
        out[i] = q[i] < 0 ? -mag : mag;
    }
}

/* The quantised linear layer: Y[b][n] = sum_k X[b][k] * What[n][k] in fp64,
 * plus A[b][n] = sum_k |X[b][k] * What[n][k]| (the scale of the rounding
 * error allowed to a lower-precision evaluation).  Output entries are
 * independent, so they may be computed by several threads; each sum runs
 * over k in order. */
void oracle_linear(const double* X, int64_t B, const double* What, int64_t N, int64_t K,
                   double* Y, double* A, int nthreads)
{
#ifdef _OPENMP
    if (nthreads > 0) omp_set_num_threads(nthreads);
#pragma omp parallel for schedule(static)
#endif
    for (int64_t n = 0; n < N; ++n) {
        const double* wr = What + n * K;
        for (int64_t b = 0; b < B; ++b) {
            const double* xr = X + b * K;
            double acc = 0.0, mag = 0.0;
            for (int64_t k = 0; k < K; ++k) {
                double p = xr[k] * wr[k];
                acc += p;
                mag += fabs(p);
            }
            Y[b * N + n] = acc;
            if (A) A[b * N + n] = mag;
        }
    }
    (void)nthreads;
}

/* Same sum for a list of (b, n) output coordinates only, reading the
 * weights straight from packed codes (used on layers too large to
 * dequantise whole).  table as in oracle_dequant. */
void oracle_linear_sampled(const double* X, int64_t K, const uint8_t* packed, int bits,
                           const oracle_codebook* cb, int table,
                           const int64_t* bs, const int64_t* ns, int64_t count,
                           double* Y, double* A, int nthreads)
{
    int64_t rb = oracle_packed_row_bytes(K, bits);
#ifdef _OPENMP
    if (nthreads > 0) omp_set_num_threads(nthreads);
#pragma omp parallel for schedule(dynamic, 16)
#endif
    for (int64_t i = 0; i < count; ++i) {
        int8_t* qrow = (int8_t*)malloc((size_t)K);
        double* wrow = (double*)malloc(sizeof(double) * (size_t)K);
        oracle_unpack(packed + ns[i] * rb, 1, K, bits, qrow);
        oracle_dequant(qrow, K, cb, table, wrow);
        const double* xr = X + bs[i] * K;
        double acc = 0.0, mag = 0.0;
        for (int64_t k = 0; k < K; ++k) {
            double p = xr[k] * wrow[k];
            acc += p;
            mag += fabs(p);
        }
        Y[i] = acc;
        if (A) A[i] = mag;
        free(qrow);
        free(wrow);
    }
    (void)nthreads;
}

/* ---- Sec. 3.2 and Eq. (3): range and base from the weights ---------- */

static int cmp_double(const void* a, const void* b)
{
    double x = *(const double*)a, y = *(const double*)b;
    return (x > y) - (x < y);
}

/* Eq. (5): the smallest t among the magnitudes |w_i| such that the energy
 * of all weights with |w_i| <= t is at least eps of the total energy.
 * Returns -1 on an empty or all-zero input or eps outside (0, 1]. */
double oracle_energy_wmin(const float* w, int64_t n, double eps)
{
    if (n <= 0 || !(eps > 0.0) || eps > 1.0) return -1.0;
    double* a = (double*)malloc(sizeof(double) * (size_t)n);
    double total = 0.0;
    for (int64_t i = 0; i < n; ++i) { a[i] = fabs((double)w[i]); total += a[i] * a[i]; }
    if (total == 0.0) { free(a); return -1.0; }
    qsort(a, (size_t)n, sizeof(double), cmp_double);
    double cum = 0.0, res = a[n - 1];
    for (int64_t i = 0; i < n; ++i) {
        cum += a[i] * a[i];
        /* all entries equal to a[i] are included at threshold t = a[i] */
        if (i + 1 < n && a[i + 1] == a[i]) continue;
        if (cum / total >= eps) { res = a[i]; break; }
    }
    free(a);
    return res;
}

/* Eq. (3): b = (w_max / w_min)^(1 / q_max). */
double oracle_base_from_range(double wmax, double wmin, int bits)
{
    int qmax = (1 << (bits - 1)) - 1;
    if (!(wmax > 0.0) || !(wmin > 0.0) || qmax < 1) return -1.0;
    return pow(wmax / wmin, 1.0 / (double)qmax);
}

/* ---- GPTQ with the Log_b quantiser (Sec. 3.3 uses GPTQ for calibration) --- */
/*
 * The published GPTQ procedure, column by column in fp64:
 *   Hd = H + damp * mean(diag H) * I   (a zero diagonal entry becomes 1 and its
 *        weight column 0: the column never sees input),
 *   Hd^-1 = U^T U with U upper triangular (Cholesky of the inverse),
 *   for j = 0 .. K-1:  q_j = Quant(w_j) (decision boundaries, R3),
 *                      e_j = (w_j - level32(q_j)) / U_jj,
 *                      w_c -= e_j * U_jc  for every later column c.
 * w_at[r][j] receives the value of w_j when column j was quantised.  The
 * quantiser's value for the error is the fp32 level (R5).  Returns 0 on
 * success, 1 when Hd is not positive definite.
 */
static int chol_lower(double* A, int64_t n)          /* A = L L^T in place (lower) */
{
    for (int64_t j = 0; j < n; ++j) {
        double d = A[j * n + j];
        for (int64_t k = 0; k < j; ++k) d -= A[j * n + k] * A[j * n + k];
        if (!(d > 0.0)) return 1;
        d = sqrt(d);
        A[j * n + j] = d;
        for (int64_t i = j + 1; i < n; ++i) {
            double s = A[i * n + j];
            for (int64_t k = 0; k < j; ++k) s -= A[i * n + k] * A[j * n + k];
            A[i * n + j] = s / d;
        }
        for (int64_t i = 0; i < j; ++i) A[i * n + j] = 0.0;
    }
    return 0;
}

/* The factor GPTQ compensates with: Hd = H + damp * mean(diag H) * I, a zero
 * diagonal entry of H (an input that never fires) first set to 1; U = the upper
 * Cholesky factor of Hd^-1 (Hd^-1 = U^T U), fp64 [K][K] row-major, zero below
 * the diagonal.  Route: Hd = L L^T, Hd^-1 by forward and backward substitution
 * on the unit columns, then the Cholesky factor of Hd^-1.  Returns 1 if Hd is
 * not positive definite. */
int oracle_gptq_factor(const double* H, int64_t K, double damp, double* U)
{
    double* A = (double*)malloc(sizeof(double) * (size_t)(K * K));
    double* Hinv = (double*)malloc(sizeof(double) * (size_t)(K * K));
    int rc = 1;
    double mean = 0.0;
    for (int64_t j = 0; j < K; ++j) mean += H[j * K + j];
    mean /= (double)K;
    memcpy(A, H, sizeof(double) * (size_t)(K * K));
    for (int64_t j = 0; j < K; ++j) {
        if (H[j * K + j] == 0.0) A[j * K + j] = 1.0;
        A[j * K + j] += damp * mean;
    }
    /* Hd = L L^T; Hd^-1 column by column from L y = e_c, L^T x = y */
    if (chol_lower(A, K)) goto out;
    for (int64_t c = 0; c < K; ++c) {
        for (int64_t i = 0; i < K; ++i) {                 /* forward */
            double s = (i == c) ? 1.0 : 0.0;
            for (int64_t k = 0; k < i; ++k) s -= A[i * K + k] * Hinv[k * K + c];
            Hinv[i * K + c] = s / A[i * K + i];
        }
        for (int64_t i = K - 1; i >= 0; --i) {            /* backward */
            double s = Hinv[i * K + c];
            for (int64_t k = i + 1; k < K; ++k) s -= A[k * K + i] * Hinv[k * K + c];
            Hinv[i * K + c] = s / A[i * K + i];
        }
    }
    /* Hd^-1 = U^T U: U = (lower Cholesky factor of Hd^-1)^T */
    if (chol_lower(Hinv, K)) goto out;
    for (int64_t j = 0; j < K; ++j)
        for (int64_t c = 0; c < K; ++c) U[j * K + c] = c >= j ? Hinv[c * K + j] : 0.0;
    rc = 0;
out:
    free(A);
    free(Hinv);
    return rc;
}

int oracle_gptq(const float* W, int64_t N, int64_t K, const double* H, double damp,
                const oracle_codebook* cb, int8_t* q, double* w_at)
{
    double* Uf = (double*)malloc(sizeof(double) * (size_t)(K * K));
    double* w = (double*)malloc(sizeof(double) * (size_t)(N * K));
    int rc = 1;
    for (int64_t i = 0; i < N * K; ++i) w[i] = (double)W[i];
    for (int64_t j = 0; j < K; ++j)                       /* a dead input's weights are dropped */
        if (H[j * K + j] == 0.0)
            for (int64_t r = 0; r < N; ++r) w[r * K + j] = 0.0;
    if (oracle_gptq_factor(H, K, damp, Uf)) goto out;
    for (int64_t r = 0; r < N; ++r) {
        double* wr = w + r * K;
        for (int64_t j = 0; j < K; ++j) {
            double x = wr[j];
            if (w_at) w_at[r * K + j] = x;
            double a = fabs(x);
            int m = 0;
            for (int t = 0; t < cb->qmax; ++t)
                if (a >= cb->tau[t]) m++;
            int8_t qv = (int8_t)(x < 0 ? -m : m);
            q[r * K + j] = qv;
            double deq = (qv < 0 ? -1.0 : 1.0) * (double)cb->level32[m];
            if (m == 0) deq = 0.0;
            double e = (x - deq) / Uf[j * K + j];
            for (int64_t c = j + 1; c < K; ++c) wr[c] -= e * Uf[j * K + c];
        }
    }
    rc = 0;
out:
    free(Uf);
    free(w);
    return rc;
}
