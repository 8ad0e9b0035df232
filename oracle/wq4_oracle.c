/*
 * wq4_oracle.c -- reference oracle for the 4-bit weight-streaming GEMV.
 *
 * TEST INFRASTRUCTURE ONLY.  This file is the plain, slow, single-threaded
 * fp64 CPU definition that the CUDA path is checked against.  Only the test
 * suite, the smoke check and the benchmark's CPU-baseline leg may load it;
 * the product library never links or calls it, and it shares no code,
 * header or table with the CUDA sources.
 *
 * What is computed (the decode-time projection of a 4-bit quantized model;
 * the paper evaluates decoding of 4-bit quantized models, Section 3 and
 * Table 1, and weights are converted offline into an artifact, Section 2.3):
 *
 *   packed weights  W  : uint32 [N][K/8]; code k of row n is the 4-bit field
 *                        at bits [4*(k%8), 4*(k%8)+4) of word W[n][k/8]
 *                        (lowest nibble first);
 *   scales          s  : fp16   [N][K/32]; one scale per group of 32 codes;
 *   dequantized     w(n,k) = (q(n,k) - 7) * s(n, k/32)       (zero point 7);
 *   activations     x  : fp16   [batch][K];
 *   output          y(b,n) = r_b * sum_{k=0}^{K-1} w(n,k) * x(b,k),
 *                   summed in fp64 in increasing k; r_b = 1 unless an RMS
 *                   factor is given (the fused RMS-norm projection below);
 *   magnitude       A(b,n) = r_b * sum_k |w(n,k) * x(b,k)|;
 *   fp16 output     fp16_RNE(y).
 *
 * The paper itself does not fix the 4-bit format (it says only "4-bit
 * quantized", Section 1 and Section 3); the layout above is this library's
 * format and is the one the CUDA path implements.
 *
 * Every function here follows its definition literally: no blocking, no
 * fusion, no reordering.  fp16 is decoded and encoded by bit manipulation
 * written out below (IEEE 754 binary16, round to nearest, ties to even).
 */
#include <math.h>
#include <stdint.h>
#include <string.h>

#define WQ4O_EXPORT __attribute__((visibility("default")))

/* ---------------------------------------------------------------- fp16 -- */

/* binary16 -> double, exact (every binary16 value is a double). */
WQ4O_EXPORT double wq4o_half_to_double(uint16_t h)
{
    int sign = (h >> 15) & 1;
    int exp = (h >> 10) & 0x1f;
    int man = h & 0x3ff;
    double v;
    if (exp == 0) {
        v = ldexp((double)man, -24);                 /* zero / subnormal */
    } else if (exp == 31) {
        v = man ? NAN : INFINITY;                    /* inf / nan */
    } else {
        v = ldexp((double)(1024 + man), exp - 25);   /* normal */
    }
    return sign ? -v : v;
}

/* double -> binary16, round to nearest, ties to even.  Overflow gives inf. */
WQ4O_EXPORT uint16_t wq4o_double_to_half(double v)
{
    uint16_t sign = signbit(v) ? 0x8000 : 0;
    double a = fabs(v);
    if (isnan(v)) return 0x7e00;
    if (a == 0.0) return sign;
    if (a < ldexp(1.0, -14)) {
        /* subnormal range: integer multiple of 2^-24, rounded half-even */
        double m = nearbyint(ldexp(a, 24));          /* default mode: ties-even */
        return (uint16_t)(sign | (uint16_t)m);       /* m == 1024 is 2^-14: ok */
    }
    int e;
    double f = frexp(a, &e);                         /* a = f * 2^e, f in [0.5,1) */
    int ex = e - 1;                                  /* a = (2f) * 2^ex */
    double m = nearbyint(ldexp(f, 11));              /* 2f * 1024, in [1024,2048] */
    if (m == 2048.0) { m = 1024.0; ex += 1; }
    if (ex > 15) return (uint16_t)(sign | 0x7c00);   /* overflow -> inf */
    return (uint16_t)(sign | ((uint16_t)(ex + 15) << 10) | (uint16_t)((int)m - 1024));
}

WQ4O_EXPORT void wq4o_half_to_double_array(const uint16_t* h, double* out, int64_t n)
{
    for (int64_t i = 0; i < n; ++i) out[i] = wq4o_half_to_double(h[i]);
}

WQ4O_EXPORT void wq4o_double_to_half_array(const double* v, uint16_t* out, int64_t n)
{
    for (int64_t i = 0; i < n; ++i) out[i] = wq4o_double_to_half(v[i]);
}

/* Spacing of binary16 numbers at |v|: 2^(floor(log2|v|) - 10) in the normal
 * range, 2^-24 below 2^-14 (including v == 0). */
WQ4O_EXPORT double wq4o_ulp16(double v)
{
    double a = fabs(v);
    if (a < ldexp(1.0, -14)) return ldexp(1.0, -24);
    int e;
    frexp(a, &e);                                    /* a in [2^(e-1), 2^e) */
    return ldexp(1.0, (e - 1) - 10);
}

/* ------------------------------------------------------------ the format -- */

/* Code k of row n: the nibble at bits [4*(k%8), 4*(k%8)+4) of W[n][k/8]. */
WQ4O_EXPORT int wq4o_code(const uint32_t* W, int K, int n, int k)
{
    uint32_t word = W[(int64_t)n * (K / 8) + k / 8];
    return (int)((word >> (4 * (k % 8))) & 0xFu);
}

/* Pack codes q[N][K] (values 0..15) into W[N][K/8]. */
WQ4O_EXPORT void wq4o_pack(const uint8_t* q, uint32_t* W, int N, int K)
{
    for (int n = 0; n < N; ++n) {
        for (int j = 0; j < K / 8; ++j) {
            uint32_t word = 0;
            for (int i = 0; i < 8; ++i) {
                uint32_t code = q[(int64_t)n * K + 8 * j + i] & 0xFu;
                word |= code << (4 * i);
            }
            W[(int64_t)n * (K / 8) + j] = word;
        }
    }
}

/* Unpack: q_out[N][K] codes and w_out[N][K] = (q - 7) * s in fp64 (exact).
 * Either output may be NULL. */
WQ4O_EXPORT void wq4o_unpack(const uint32_t* W, const uint16_t* s, int N, int K,
                             uint8_t* q_out, double* w_out)
{
    for (int n = 0; n < N; ++n) {
        for (int k = 0; k < K; ++k) {
            int q = wq4o_code(W, K, n, k);
            if (q_out) q_out[(int64_t)n * K + k] = (uint8_t)q;
            if (w_out) {
                double sc = wq4o_half_to_double(s[(int64_t)n * (K / 32) + k / 32]);
                w_out[(int64_t)n * K + k] = (double)(q - 7) * sc;
            }
        }
    }
}

/* ------------------------------------------------------------------ GEMV -- */

/* y[b][n] = r_b * sum_k w(n,k) x(b,k) in fp64, increasing k.
 *   W    : uint32 [N][K/8]     s : fp16 [N][K/32]     x : fp16 [batch][K]
 *   r    : double [batch] RMS factors, or NULL for r_b = 1
 *   y    : double [batch][N]   A : double [batch][N]   y16 : fp16 [batch][N]
 * Any of y, A, y16 may be NULL. */
WQ4O_EXPORT void wq4o_gemv(const uint32_t* W, const uint16_t* s, const uint16_t* x,
                           int N, int K, int batch, const double* r,
                           double* y, double* A, uint16_t* y16)
{
    for (int b = 0; b < batch; ++b) {
        double rb = r ? r[b] : 1.0;
        for (int n = 0; n < N; ++n) {
            double acc = 0.0, mag = 0.0;
            for (int k = 0; k < K; ++k) {
                int q = wq4o_code(W, K, n, k);
                double sc = wq4o_half_to_double(s[(int64_t)n * (K / 32) + k / 32]);
                double w = (double)(q - 7) * sc;
                double xv = wq4o_half_to_double(x[(int64_t)b * K + k]);
                acc += w * xv;
                mag += fabs(w * xv);
            }
            acc *= rb;
            mag *= rb;
            if (y) y[(int64_t)b * N + n] = acc;
            if (A) A[(int64_t)b * N + n] = mag;
            if (y16) y16[(int64_t)b * N + n] = wq4o_double_to_half(acc);
        }
    }
}

/* ------------------------------------------------------ decode-chain glue -- */
/*
 * The glue between projections of one decoded token: RMS normalisation
 * without a learned gain, SiLU(gate) * up, and residual adds.  The paper's
 * compiler fuses such operators into the kernels ("kernel fusion",
 * Section 2.3); the oracle keeps each one separate and literal.
 */

/* r = 1 / sqrt(mean(v^2) + eps) over v[0..n), v in fp16. */
WQ4O_EXPORT double wq4o_rms_factor(const uint16_t* v, int n, double eps)
{
    double ss = 0.0;
    for (int i = 0; i < n; ++i) {
        double t = wq4o_half_to_double(v[i]);
        ss += t * t;
    }
    return 1.0 / sqrt(ss / (double)n + eps);
}

/* v[i] = fp16_RNE(r * u[i]) with r = 1 / sqrt(mean(u^2) + eps): the RMS
 * normalisation (no learned gain) that turns a layer's output into the next
 * layer's input. */
WQ4O_EXPORT void wq4o_rms_normalize(const uint16_t* u, int n, double eps, uint16_t* v)
{
    double r = wq4o_rms_factor(u, n, eps);
    for (int i = 0; i < n; ++i) v[i] = wq4o_double_to_half(r * wq4o_half_to_double(u[i]));
}

/* m[i] = silu(g[i]) * u[i] with silu(t) = t / (1 + exp(-t)); fp64 result
 * and its fp16 rounding (either output may be NULL). */
WQ4O_EXPORT void wq4o_silu_mul(const uint16_t* g, const uint16_t* u, int n,
                               double* m, uint16_t* m16)
{
    for (int i = 0; i < n; ++i) {
        double gv = wq4o_half_to_double(g[i]);
        double uv = wq4o_half_to_double(u[i]);
        double v = gv / (1.0 + exp(-gv)) * uv;
        if (m) m[i] = v;
        if (m16) m16[i] = wq4o_double_to_half(v);
    }
}

/* z[i] = fp16_RNE(a[i] + b[i]); the fp64 sum of two binary16 values is exact. */
WQ4O_EXPORT void wq4o_add_fp16(const uint16_t* a, const uint16_t* b, int n, uint16_t* z)
{
    for (int i = 0; i < n; ++i)
        z[i] = wq4o_double_to_half(wq4o_half_to_double(a[i]) + wq4o_half_to_double(b[i]));
}
