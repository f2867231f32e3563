/*
 * puro_oracle.c -- plain, slow, CPU reference ("oracle") for the FP8 linear
 * training path of Puro-2B.
 *
 * TEST INFRASTRUCTURE ONLY.  Nothing in the product path may link, load or
 * call this file; only the test suite, the smoke check and the CPU-baseline
 * leg of the benchmark do.  It shares no code, header, table or constant
 * generator with the CUDA library.
 *
 * What it computes, and where the paper defines it:
 *   - FP8 operands are E4M3 for every linear-layer GEMM (paper, section
 *     "FP8 Mixed-Precision Training"; appendix "Production Training Details",
 *     paragraph "FP8 implementation pipeline" and the precision-flow figure).
 *     E5M2 is implemented as the contrasted format of the same section.
 *     Format parameters follow the OCP FP8 formats paper cited there
 *     (Micikevicius et al. 2022, Table 1): E4M3 bias 7, max 448, no infinity,
 *     NaN = S.1111.111; E5M2 bias 15, max 57344, infinities S.11111.00.
 *   - Scales are computed online per local group: activations and their
 *     gradients use 1x128 groups along the GEMM reduction dimension, weights
 *     use 128x128 blocks (section "FP8 Mixed-Precision Training").
 *   - Each group scale is a power of two (E8M0 expressiveness), same section.
 *     Reading taken where the paper is silent: the scale is the smallest power
 *     of two s with amax/s <= format max, so no value saturates.
 *   - Fprop Y = X W^T, Dgrad dX = dY W, Wgrad dW = dY^T X, all three from FP8
 *     operands, BF16 output (same section, "FP8 implementation pipeline").
 *     Here every product is formed from the dequantised operands and summed
 *     in fp64, in plain k order.
 *   - Per-tensor current scaling (the contrast drawn in the same section:
 *     a single scale per tensor): scale = fp32(fmt_max / amax),
 *     codes = RNE_sat(fp32(x * scale)), scale_inv = fp32(1 / scale).
 *   - RMSNorm ahead of the quantiser (the model's normalisation before the
 *     attention and MLP projections, section "Model architecture and
 *     pretraining system": the Qwen3 architecture): rstd = 1/sqrt(mean h^2
 *     + eps) per row, y = bf16((h * rstd) * gamma).
 *   - SwiGLU ahead of the quantiser (the same architecture's MLP: the down
 *     projection receives silu(gate) * up): h = bf16(g * u / (1 + e^-g)).
 *   - The MuonH hyperball step (section "Hyperball Optimization", Eq.
 *     hyperball-update): u_hat = u / ||u||_F, W~ = W - eta R u_hat,
 *     W <- R W~ / ||W~||_F with R = ||W_0||_F fixed.
 *
 * Build: gcc -std=c11 -O2 -ffp-contract=off -fPIC -shared -pthread.
 * No fast-math: every float/double operation below is an IEEE operation in
 * round-to-nearest-even.
 */
#include <float.h>
#include <math.h>
#include <pthread.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define ORACLE_E4M3 0
#define ORACLE_E5M2 1

/* ---------------------------------------------------------------------- */
/* FP8 formats (OCP FP8, Table 1 of the cited formats paper).             */
/* ---------------------------------------------------------------------- */
typedef struct {
    int man_bits;      /* explicit mantissa bits */
    int exp_bits;      /* exponent field width */
    int bias;          /* exponent bias */
    double max;        /* largest finite magnitude */
    uint8_t max_code;  /* code of +max */
    uint8_t nan_code;  /* canonical positive NaN */
} fp8_format;

static const fp8_format FORMATS[2] = {
    /* E4M3: 1.110 x 2^8 = 448, code 0x7E; NaN 0x7F; no infinities. */
    {3, 4, 7, 448.0, 0x7E, 0x7F},
    /* E5M2: 1.11 x 2^15 = 57344, code 0x7B; +inf 0x7C; NaN 0x7D..0x7F. */
    {2, 5, 15, 57344.0, 0x7B, 0x7F},
};

double oracle_fmt_max(int fmt) { return FORMATS[fmt].max; }

/* Value of an FP8 code, exactly, as a double. */
double oracle_fp8_decode(uint8_t code, int fmt)
{
    const fp8_format *f = &FORMATS[fmt];
    int sign = code >> 7;
    int e = (code >> f->man_bits) & ((1 << f->exp_bits) - 1);
    int m = code & ((1 << f->man_bits) - 1);
    int emax_field = (1 << f->exp_bits) - 1;
    double v;
    if (fmt == ORACLE_E4M3 && e == emax_field && m == (1 << f->man_bits) - 1)
        return NAN;                                   /* S.1111.111 */
    if (fmt == ORACLE_E5M2 && e == emax_field) {
        if (m != 0) return NAN;                       /* S.11111.{01,10,11} */
        v = INFINITY;                                 /* S.11111.00 */
    } else if (e == 0) {
        /* subnormal: m * 2^(1 - bias - man_bits) */
        v = ldexp((double)m, 1 - f->bias - f->man_bits);
    } else {
        /* normal: (2^man_bits + m) * 2^(e - bias - man_bits) */
        v = ldexp((double)((1 << f->man_bits) + m), e - f->bias - f->man_bits);
    }
    return sign ? -v : v;
}

/*
 * Round-to-nearest-even with saturation to the largest finite value
 * ("satfinite"): NaN -> canonical NaN; |v| >= max (including infinity)
 * -> +-max; otherwise the nearest representable value, ties to the code
 * with an even mantissa.  The sign is always kept, so a negative value
 * that rounds to zero gives -0 (0x80).
 */
uint8_t oracle_fp8_encode(double v, int fmt)
{
    const fp8_format *f = &FORMATS[fmt];
    if (isnan(v)) return f->nan_code;
    uint8_t sign = signbit(v) ? 0x80 : 0x00;
    double a = fabs(v);
    if (a >= f->max) return sign | f->max_code;

    int emin = 1 - f->bias;          /* exponent of the smallest normal */
    int e = emin;
    if (a != 0.0) {
        int fe;
        frexp(a, &fe);               /* a in [2^(fe-1), 2^fe) */
        e = fe - 1;
        if (e < emin) e = emin;      /* subnormals share the min-normal quantum */
    }
    /* spacing of representable values in [2^e, 2^(e+1)) */
    double quantum = ldexp(1.0, e - f->man_bits);
    /* a / quantum is an exact power-of-two scaling; nearbyint() rounds
     * half to even in the default rounding mode. */
    double r = nearbyint(a / quantum) * quantum;

    if (r == 0.0) return sign;
    int field, mant;
    if (r < ldexp(1.0, emin)) {
        field = 0;
        mant = (int)(r / ldexp(1.0, emin - f->man_bits));
    } else {
        int fe;
        frexp(r, &fe);
        int er = fe - 1;                              /* r in [2^er, 2^(er+1)) */
        field = er + f->bias;
        mant = (int)(r / ldexp(1.0, er - f->man_bits)) - (1 << f->man_bits);
    }
    return sign | (uint8_t)((field << f->man_bits) | mant);
}

/* ---------------------------------------------------------------------- */
/* BF16 helpers                                                            */
/* ---------------------------------------------------------------------- */
static double bf16_to_double(uint16_t bits)
{
    uint32_t u = (uint32_t)bits << 16;
    float f;
    memcpy(&f, &u, sizeof f);
    return (double)f;
}

static float bf16_to_float(uint16_t bits)
{
    uint32_t u = (uint32_t)bits << 16;
    float f;
    memcpy(&f, &u, sizeof f);
    return f;
}

/* Round a double to the nearest bf16 (ties to even); NaN -> 0x7FC0. */
uint16_t oracle_bf16_from_double(double v)
{
    if (isnan(v)) return 0x7FC0;
    uint16_t sign = signbit(v) ? 0x8000 : 0;
    double a = fabs(v);
    if (a == 0.0) return sign;
    /* bf16: 8 exponent bits (bias 127), 7 mantissa bits; min normal 2^-126,
     * subnormal quantum 2^-133.  Rounded once, directly from the double. */
    int fe;
    frexp(a, &fe);
    int e = fe - 1;
    if (e < -126) e = -126;
    double quantum = ldexp(1.0, e - 7);
    double r = nearbyint(a / quantum) * quantum;
    if (r >= ldexp(1.0, 128)) return sign | 0x7F80;  /* overflow -> inf */
    if (r == 0.0) return sign;
    if (r < ldexp(1.0, -126)) return sign | (uint16_t)(r / ldexp(1.0, -133));
    frexp(r, &fe);
    int er = fe - 1;
    int mant = (int)(r / ldexp(1.0, er - 7)) - 128;
    return sign | (uint16_t)(((er + 127) << 7) | mant);
}

/* ---------------------------------------------------------------------- */
/* amax                                                                    */
/* ---------------------------------------------------------------------- */
/*
 * max |x| over n bf16 values, returned as bf16 bits.  Comparing the bit
 * patterns with the sign cleared is the exact order of magnitudes for
 * finite values; infinity (0x7F80) sorts above every finite value and NaN
 * (> 0x7F80) above infinity, so a NaN anywhere gives a NaN amax.
 */
uint16_t oracle_amax_bf16(const uint16_t *x, int64_t n)
{
    uint16_t m = 0;
    for (int64_t i = 0; i < n; ++i) {
        uint16_t a = x[i] & 0x7FFF;
        if (a > m) m = a;
    }
    return m;
}

/* ---------------------------------------------------------------------- */
/* Power-of-two (E8M0) group scale                                         */
/* ---------------------------------------------------------------------- */
/*
 * The biased exponent g of the group scale s = 2^(g-127):
 *   amax == 0          -> g = 127 (s = 1)
 *   amax not finite    -> g = 0xFF (the E8M0 NaN)
 *   otherwise          -> g = clamp(k + 127, 0, 254) with k the smallest
 *                         integer such that amax <= fmt_max * 2^k.
 * The comparison is exact in double (fmt_max * 2^k is exact).
 */
uint8_t oracle_e8m0_from_amax(uint16_t amax_bits, int fmt)
{
    double a = bf16_to_double(amax_bits);
    if (a == 0.0) return 127;
    if (!isfinite(a)) return 0xFF;
    double fmax = FORMATS[fmt].max;
    int fe;
    frexp(a, &fe);                     /* a >= 2^(fe-1) */
    int k = (fe - 1) - 17;             /* fmax * 2^k < 2^16 * 2^(fe-18) < a */
    while (!(a <= ldexp(fmax, k))) ++k;
    int g = k + 127;
    if (g < 0) g = 0;
    if (g > 254) g = 254;
    return (uint8_t)g;
}

/* Code for element x of a group with scale exponent g (the group rule). */
static uint8_t quantize_in_group(uint16_t xbits, uint8_t g, int fmt)
{
    if (g == 0xFF) /* non-finite group: every code is NaN, sign kept */
        return (uint8_t)((xbits & 0x8000 ? 0x80 : 0x00) | FORMATS[fmt].nan_code);
    /* x / s = x * 2^(127 - g), exact in double */
    return oracle_fp8_encode(bf16_to_double(xbits) * ldexp(1.0, 127 - (int)g), fmt);
}

/*
 * 1x128 groups along each row (the reduction dimension of the GEMM that
 * consumes the rows).  x: [rows, cols] row-major bf16; cols % 128 == 0.
 * q: [rows, cols] codes; s: [rows, cols/128] scale exponents (row-major).
 */
void oracle_quantize_rows_1x128(const uint16_t *x, int64_t rows, int64_t cols, int fmt,
                                uint8_t *q, uint8_t *s)
{
    int64_t ng = cols / 128;
    for (int64_t r = 0; r < rows; ++r) {
        for (int64_t gi = 0; gi < ng; ++gi) {
            const uint16_t *grp = x + r * cols + gi * 128;
            uint8_t g = oracle_e8m0_from_amax(oracle_amax_bf16(grp, 128), fmt);
            s[r * ng + gi] = g;
            for (int j = 0; j < 128; ++j)
                q[r * cols + gi * 128 + j] = quantize_in_group(grp[j], g, fmt);
        }
    }
}

/*
 * 128x128 blocks (weights).  x: [rows, cols]; rows, cols % 128 == 0.
 * q: [rows, cols]; s: [rows/128, cols/128] (row-major).
 */
void oracle_quantize_blocks_128x128(const uint16_t *x, int64_t rows, int64_t cols, int fmt,
                                    uint8_t *q, uint8_t *s)
{
    int64_t nbr = rows / 128, nbc = cols / 128;
    for (int64_t br = 0; br < nbr; ++br) {
        for (int64_t bc = 0; bc < nbc; ++bc) {
            uint16_t m = 0;
            for (int64_t i = 0; i < 128; ++i) {
                uint16_t a = oracle_amax_bf16(x + (br * 128 + i) * cols + bc * 128, 128);
                if (a > m) m = a;
            }
            uint8_t g = oracle_e8m0_from_amax(m, fmt);
            s[br * nbc + bc] = g;
            for (int64_t i = 0; i < 128; ++i)
                for (int64_t j = 0; j < 128; ++j) {
                    int64_t idx = (br * 128 + i) * cols + bc * 128 + j;
                    q[idx] = quantize_in_group(x[idx], g, fmt);
                }
        }
    }
}

/*
 * Per-tensor current scaling from a given amax (bf16 bits):
 *   amax non-finite -> every code NaN (sign kept), scale_inv = NaN
 *   scale = fp32(fmt_max / amax); 1 if amax == 0; FLT_MAX if the quotient
 *           overflows to infinity
 *   code  = RNE_sat(fp32(x * scale))        (two roundings, by definition)
 *   scale_inv = fp32(1 / scale)
 */
void oracle_quantize_tensor(const uint16_t *x, int64_t n, int fmt, uint16_t amax_bits,
                            uint8_t *q, float *scale_inv)
{
    if ((amax_bits & 0x7FFF) >= 0x7F80) {
        for (int64_t i = 0; i < n; ++i)
            q[i] = (uint8_t)((x[i] & 0x8000 ? 0x80 : 0x00) | FORMATS[fmt].nan_code);
        *scale_inv = NAN;
        return;
    }
    float amax = bf16_to_float(amax_bits);
    float scale = 1.0f;
    if (amax != 0.0f) {
        scale = (float)FORMATS[fmt].max / amax;
        if (isinf(scale)) scale = FLT_MAX;
    }
    for (int64_t i = 0; i < n; ++i) {
        float p = bf16_to_float(x[i]) * scale;
        q[i] = oracle_fp8_encode((double)p, fmt);
    }
    *scale_inv = 1.0f / scale;
}

/* ---------------------------------------------------------------------- */
/* Dequantisation to double                                                */
/* ---------------------------------------------------------------------- */
static double e8m0_value(uint8_t g)
{
    if (g == 0xFF) return NAN;
    return ldexp(1.0, (int)g - 127);
}

/* out[r, c] = decode(q[r, c]) * 2^(s[r, c/128] - 127); s is [rows, cols/128]. */
void oracle_dequant_rows_1x128(const uint8_t *q, const uint8_t *s, int64_t rows, int64_t cols,
                               int fmt, double *out)
{
    int64_t ng = cols / 128;
    for (int64_t r = 0; r < rows; ++r)
        for (int64_t c = 0; c < cols; ++c)
            out[r * cols + c] = oracle_fp8_decode(q[r * cols + c], fmt) * e8m0_value(s[r * ng + c / 128]);
}

/* out[r, c] = decode(q[r, c]) * 2^(s[r/128, c/128] - 127). */
void oracle_dequant_blocks_128x128(const uint8_t *q, const uint8_t *s, int64_t rows, int64_t cols,
                                   int fmt, double *out)
{
    int64_t nbc = cols / 128;
    for (int64_t r = 0; r < rows; ++r)
        for (int64_t c = 0; c < cols; ++c)
            out[r * cols + c] = oracle_fp8_decode(q[r * cols + c], fmt) *
                                e8m0_value(s[(r / 128) * nbc + c / 128]);
}

/* out[i] = decode(q[i]) * scale_inv. */
void oracle_dequant_tensor(const uint8_t *q, int64_t n, int fmt, float scale_inv, double *out)
{
    for (int64_t i = 0; i < n; ++i)
        out[i] = oracle_fp8_decode(q[i], fmt) * (double)scale_inv;
}

/* out[i] = value of bf16 x[i]. */
void oracle_bf16_to_double(const uint16_t *x, int64_t n, double *out)
{
    for (int64_t i = 0; i < n; ++i) out[i] = bf16_to_double(x[i]);
}

/* ---------------------------------------------------------------------- */
/* GEMM: out[m, n] = sum_k a[m, k] * b[n, k], fp64, plain k order          */
/* ---------------------------------------------------------------------- */
typedef struct {
    const double *a, *b;
    double *out;
    int64_t M, N, K, m0, m1;
} gemm_job;

static void *gemm_worker(void *p)
{
    gemm_job *j = (gemm_job *)p;
    for (int64_t m = j->m0; m < j->m1; ++m)
        for (int64_t n = 0; n < j->N; ++n) {
            double acc = 0.0;
            for (int64_t k = 0; k < j->K; ++k) acc += j->a[m * j->K + k] * j->b[n * j->K + k];
            j->out[m * j->N + n] = acc;
        }
    return NULL;
}

/*
 * a: [M, K], b: [N, K] (both row-major, reduction along the rows), out: [M, N].
 * fprop:  a = X,   b = W     (Y  = X W^T)
 * dgrad:  a = dY,  b = W^T   (dX = dY W)
 * wgrad:  a = dY^T, b = X^T  (dW = dY^T X)
 * nthreads > 1 splits the rows of out across POSIX threads; each output is
 * still one sequential fp64 sum.
 */
int oracle_gemm_tn(const double *a, const double *b, int64_t M, int64_t N, int64_t K,
                   double *out, int nthreads)
{
    if (nthreads < 1) nthreads = 1;
    if (M < 1) return 0;
    if (nthreads > M) nthreads = (int)M;
    pthread_t *th = (pthread_t *)malloc(sizeof(pthread_t) * (size_t)nthreads);
    gemm_job *jobs = (gemm_job *)malloc(sizeof(gemm_job) * (size_t)nthreads);
    char *running = (char *)calloc((size_t)nthreads, 1);
    if (!th || !jobs || !running) { free(th); free(jobs); free(running); return -1; }
    for (int t = 0; t < nthreads; ++t) {
        jobs[t] = (gemm_job){a, b, out, M, N, K, M * t / nthreads, M * (t + 1) / nthreads};
        if (t > 0 && pthread_create(&th[t], NULL, gemm_worker, &jobs[t]) == 0) running[t] = 1;
        else if (t > 0) gemm_worker(&jobs[t]);
    }
    gemm_worker(&jobs[0]);
    for (int t = 1; t < nthreads; ++t)
        if (running[t]) pthread_join(th[t], NULL);
    free(th);
    free(jobs);
    free(running);
    return 0;
}

/* out[i] = sum_k a[ai[i], k] * b[bi[i], k] for a list of (row of a, row of b) pairs. */
void oracle_dot_pairs(const double *a, const double *b, int64_t K, const int64_t *ai,
                      const int64_t *bi, int64_t npairs, double *out)
{
    for (int64_t i = 0; i < npairs; ++i) {
        double acc = 0.0;
        const double *ra = a + ai[i] * K, *rb = b + bi[i] * K;
        for (int64_t k = 0; k < K; ++k) acc += ra[k] * rb[k];
        out[i] = acc;
    }
}

/* ---------------------------------------------------------------------- */
/* Elementwise array forms of the codec (for the test harness)             */
/* ---------------------------------------------------------------------- */
void oracle_fp8_decode_array(const uint8_t *q, int64_t n, int fmt, double *out)
{
    for (int64_t i = 0; i < n; ++i) out[i] = oracle_fp8_decode(q[i], fmt);
}

void oracle_fp8_encode_array(const double *v, int64_t n, int fmt, uint8_t *out)
{
    for (int64_t i = 0; i < n; ++i) out[i] = oracle_fp8_encode(v[i], fmt);
}

void oracle_bf16_from_double_array(const double *v, int64_t n, uint16_t *out)
{
    for (int64_t i = 0; i < n; ++i) out[i] = oracle_bf16_from_double(v[i]);
}

void oracle_e8m0_from_amax_array(const uint16_t *amax_bits, int64_t n, int fmt, uint8_t *out)
{
    for (int64_t i = 0; i < n; ++i) out[i] = oracle_e8m0_from_amax(amax_bits[i], fmt);
}

/* ---------------------------------------------------------------------- */
/* RMSNorm producer                                                        */
/* ---------------------------------------------------------------------- */
/*
 * Per-row reciprocal RMS of h [rows, cols] (bf16): rstd[r] = 1 /
 * sqrt(sum_k h[r,k]^2 / cols + eps), in fp64 (each square is exact in fp64;
 * the sum is taken in k order).
 */
void oracle_rmsnorm_rstd(const uint16_t *h, int64_t rows, int64_t cols, double eps, double *rstd)
{
    for (int64_t r = 0; r < rows; ++r) {
        double ss = 0.0;
        for (int64_t k = 0; k < cols; ++k) {
            const double v = bf16_to_double(h[r * cols + k]);
            ss += v * v;
        }
        rstd[r] = 1.0 / sqrt(ss / (double)cols + eps);
    }
}

/*
 * The normalised activation the quantiser receives, given an fp32 rstd per
 * row: y[r,k] = bf16_rne(fp32(fp32(h[r,k] * rstd[r]) * gamma[k])), the two
 * products in fp32 round-to-nearest in that order; gamma NULL means no gain
 * (the second product is skipped).
 */
void oracle_rmsnorm_apply_f32(const uint16_t *h, int64_t rows, int64_t cols, const float *rstd,
                              const uint16_t *gamma, uint16_t *y)
{
    for (int64_t r = 0; r < rows; ++r)
        for (int64_t k = 0; k < cols; ++k) {
            float p = bf16_to_float(h[r * cols + k]) * rstd[r];
            if (gamma) p = p * bf16_to_float(gamma[k]);
            y[r * cols + k] = oracle_bf16_from_double((double)p);
        }
}

/* ---------------------------------------------------------------------- */
/* SwiGLU producer                                                         */
/* ---------------------------------------------------------------------- */
/*
 * The down projection's input in the gated MLP: h[r,k] = bf16_rne(silu(g) * u)
 * with silu(g) = g / (1 + e^-g), evaluated in fp64 (libm exp) and rounded
 * once to bf16.  g and u are bf16 [rows, cols] with rows ld elements apart
 * (ld >= cols; views into the gate/up halves of one [rows, 2*cols] output
 * have ld = 2*cols); h is contiguous [rows, cols].
 */
void oracle_swiglu(const uint16_t *g, const uint16_t *u, int64_t rows, int64_t cols, int64_t ld, uint16_t *h)
{
    for (int64_t r = 0; r < rows; ++r)
        for (int64_t k = 0; k < cols; ++k) {
            const double gv = bf16_to_double(g[r * ld + k]);
            const double uv = bf16_to_double(u[r * ld + k]);
            const double silu = gv / (1.0 + exp(-gv));
            h[r * cols + k] = oracle_bf16_from_double(silu * uv);
        }
}

/* ---------------------------------------------------------------------- */
/* MuonH hyperball step                                                    */
/* ---------------------------------------------------------------------- */
/* Frobenius norm of n fp32 values, in fp64 (index order). */
double oracle_frobenius_norm(const float *x, int64_t n)
{
    double ss = 0.0;
    for (int64_t i = 0; i < n; ++i) ss += (double)x[i] * (double)x[i];
    return sqrt(ss);
}

/*
 * One hyperball update of a wrapped matrix (n values, any shape: the
 * Frobenius norm is that of the flattened matrix), in the order of the
 * equation: normalise the Muon direction, step by eta * R along it, then
 * project back onto the sphere of radius R.  w_new is fp64 (the fp32 master
 * weight the kernels write is compared against it within a tolerance).
 * Reading where the equation is undefined: a zero Muon direction (||u|| = 0)
 * takes no step (u_hat = 0), so W is only projected.
 */
void oracle_muonh_step(const float *w, const float *u, int64_t n, double eta, double radius, double *w_new)
{
    const double unorm = oracle_frobenius_norm(u, n);
    double tnorm2 = 0.0;
    for (int64_t i = 0; i < n; ++i) {
        const double u_hat = unorm > 0.0 ? (double)u[i] / unorm : 0.0;
        const double wt = (double)w[i] - eta * radius * u_hat;
        w_new[i] = wt;
        tnorm2 += wt * wt;
    }
    const double tnorm = sqrt(tnorm2);
    for (int64_t i = 0; i < n; ++i) w_new[i] = radius * (w_new[i] / tnorm);
}
