/*
 * PVS oracle, plain C.  TEST INFRASTRUCTURE ONLY: nothing in the product
 * path may link, load or call this file.  Only tests/, the smoke check and
 * the CPU-baseline leg of bench.py use it.
 *
 * What it computes (arXiv 2608.07152):
 *   - PVS per-vector Int8 quantization (Sec. 2.3.1): s_v = f32(||v||_inf/127),
 *     z_v = clip(round(v/s_v), -127, 127); a zero vector has s_v = 1, z_v = 0.
 *   - The upward-rounded Euclidean norms that the residual bound
 *     E = ||e_q|| ||v|| + ||q_hat|| ||e_v|| (Sec. 2.3.1) and the guard
 *     G = (|c| + E + ||q||_up ||v||_up) gamma_m (Appendix A.1) need.
 *   - gamma_m >= a_m / (1 - a_m), a_m = (8m + 64) * f32::EPSILON (Appendix A.1).
 *   - The interval [c - (E+G), c + (E+G)] with outward-rounded endpoints
 *     around the centre score c = s_q s_v <z_q, z_v> (Sec. 2.3.1, App. A.1).
 *
 * The paper does not fix the operation order of these bounds; the readings
 * used here (and by the product kernels, which are written separately) are:
 *   round(): half away from zero.  s_v: IEEE f32 division maxabs / 127.0f;
 *   if that underflows to 0 for a nonzero vector, the smallest positive
 *   subnormal.  v_j / s_v: IEEE f32 division.
 *   norm_bound(x) for a vector of binary64 values x_j:
 *     M = max |x_j|, M = f * 2^e with f in [0.5, 1)  (so every x_j^2 < 4^e);
 *     t_j = ceil(RU64(x_j * x_j) * 2^(48 - 2e))   (an integer <= 2^48);
 *     T = sum_j t_j  (exact integer sum, any order);
 *     norm_bound = RU32(RU_sqrt64(RU64(T) * 2^(2e - 48))), and 0 if M == 0.
 *   It is an upper bound on ||x||_2 whatever the summation order, and every
 *   step is a single IEEE operation with a stated rounding, so it is
 *   reproducible bit for bit.
 *   Interval, in f32 (RN = to nearest, RU = up, RD = down):
 *     c = RN(RN(s_q * s_v) * RN(float(dot)))
 *     E = RU(RU(enorm_q * vnorm) + RU(qhat * enorm_v))
 *     G = RU(RU(RU(|c| + E) + RU(qnorm * vnorm)) * gamma)
 *     r = RU(E + G);  lo = RD(c - r);  hi = RU(c + r)
 *
 * Directed rounding is done with fesetround around single operations on
 * volatile operands; build with -O0 -frounding-math -ffp-contract=off.
 */
#include <fenv.h>
#include <math.h>
#include <stdint.h>
#include <string.h>

#pragma STDC FENV_ACCESS ON

/* ---- single operations with a stated rounding mode ---------------------- */

static float f32_op(int mode, char op, float a, float b) {
    volatile float va = a, vb = b, r = 0.0f;
    int old = fegetround();
    fesetround(mode);
    switch (op) {
        case '+': r = va + vb; break;
        case '-': r = va - vb; break;
        case '*': r = va * vb; break;
        case '/': r = va / vb; break;
    }
    fesetround(old);
    return r;
}

static double f64_mul(int mode, double a, double b) {
    volatile double va = a, vb = b, r;
    int old = fegetround();
    fesetround(mode);
    r = va * vb;
    fesetround(old);
    return r;
}

static double f64_sqrt(int mode, double a) {
    volatile double va = a, r;
    int old = fegetround();
    fesetround(mode);
    r = sqrt(va);
    fesetround(old);
    return r;
}

static double i64_to_f64(int mode, int64_t t) {
    volatile int64_t vt = t;
    volatile double r;
    int old = fegetround();
    fesetround(mode);
    r = (double)vt;
    fesetround(old);
    return r;
}

static float f64_to_f32(int mode, double a) {
    volatile double va = a;
    volatile float r;
    int old = fegetround();
    fesetround(mode);
    r = (float)va;
    fesetround(old);
    return r;
}

/* ---- exported oracle functions ------------------------------------------- */

/* Upward-rounded Euclidean norm of m binary64 values (reading stated above). */
float orc_norm_bound(const double* x, int32_t m) {
    double M = 0.0;
    for (int32_t j = 0; j < m; ++j) {
        double a = fabs(x[j]);
        if (a > M) M = a;
    }
    if (M == 0.0) return 0.0f;
    int e;
    (void)frexp(M, &e);                       /* M = f * 2^e, f in [0.5, 1) */
    int64_t T = 0;
    for (int32_t j = 0; j < m; ++j) {
        double sq = f64_mul(FE_UPWARD, x[j], x[j]);
        double scaled = ldexp(sq, 48 - 2 * e);   /* exact power-of-two scaling */
        T += (int64_t)ceil(scaled);
    }
    double Tup = i64_to_f64(FE_UPWARD, T);
    double sumsq = ldexp(Tup, 2 * e - 48);
    double root = f64_sqrt(FE_UPWARD, sumsq);
    return f64_to_f32(FE_UPWARD, root);
}

/* gamma_m = RU(a / (1 - a)), a = (8m + 64) * 2^-23; both a and 1 - a are
 * exact in f32 for the sizes accepted (a < 1).  Returns -1 if a >= 1. */
float orc_gamma(int32_t m) {
    double a64 = (8.0 * (double)m + 64.0) * ldexp(1.0, -23);
    if (a64 >= 1.0) return -1.0f;
    float a = (float)a64;
    float den = f32_op(FE_DOWNWARD, '-', 1.0f, a);
    return f32_op(FE_UPWARD, '/', a, den);
}

static double round_half_away(double t) {
    /* t is an f32 value; t +/- 0.5 is exact in binary64 for |t| < 2^29. */
    return t >= 0.0 ? floor(t + 0.5) : -floor(-t + 0.5);
}

/* Quantize one vector.  Returns 0, or 1 if the input holds a non-finite
 * value, or 2 if a norm bound overflows f32. */
int32_t orc_quantize_one(const float* v, int32_t m, int8_t* z, float* s_out,
                         float* vnorm_out, float* enorm_out, double* scratch) {
    float maxabs = 0.0f;
    for (int32_t j = 0; j < m; ++j) {
        if (!isfinite(v[j])) return 1;
        float a = fabsf(v[j]);
        if (a > maxabs) maxabs = a;
    }
    float s;
    if (maxabs == 0.0f) {
        s = 1.0f;
        for (int32_t j = 0; j < m; ++j) z[j] = 0;
    } else {
        s = f32_op(FE_TONEAREST, '/', maxabs, 127.0f);
        if (s == 0.0f) s = ldexpf(1.0f, -149);
        for (int32_t j = 0; j < m; ++j) {
            float t = f32_op(FE_TONEAREST, '/', v[j], s);
            double r = round_half_away((double)t);
            if (r > 127.0) r = 127.0;
            if (r < -127.0) r = -127.0;
            z[j] = (int8_t)r;
        }
    }
    /* ||v||_up */
    for (int32_t j = 0; j < m; ++j) scratch[j] = (double)v[j];
    float vn = orc_norm_bound(scratch, m);
    /* e_j = v_j - s z_j is exact in binary64 (s*z_j has <= 31 significant
     * bits and the difference spans < 53 bits). */
    for (int32_t j = 0; j < m; ++j)
        scratch[j] = (double)v[j] - (double)s * (double)z[j];
    float en = orc_norm_bound(scratch, m);
    *s_out = s;
    *vnorm_out = vn;
    *enorm_out = en;
    if (isinf(vn) || isinf(en)) return 2;
    return 0;
}

/* Quantize n row-major vectors of dimension m.  Codes are written with row
 * stride ldz (>= m); columns m..ldz-1 are zeroed.  Returns the first nonzero
 * per-vector status (see orc_quantize_one), else 0. */
int32_t orc_quantize(const float* V, int64_t n, int32_t m, int8_t* Z, int32_t ldz,
                     float* s, float* vnorm, float* enorm, double* scratch) {
    int32_t status = 0;
    for (int64_t i = 0; i < n; ++i) {
        int8_t* zi = Z + i * (int64_t)ldz;
        for (int32_t j = m; j < ldz; ++j) zi[j] = 0;
        int32_t st = orc_quantize_one(V + i * (int64_t)m, m, zi, &s[i], &vnorm[i],
                                      &enorm[i], scratch);
        if (st && !status) status = st;
    }
    return status;
}

/* Scalar-quantization intervals (the ablation of Sec. 3.5 / 4.4; reading of
 * this library): one scale for the whole corpus, s = RN(max_{v,j} |v_j| /
 * 127) (1 for an all-zero corpus, the smallest subnormal if the quotient
 * underflows), the same codes, residuals and norm bounds as Sec. 2.3.1 per
 * vector with s in place of s_v.  Returns the scale, or NaN if an entry is
 * not finite. */
float orc_global_scale(const float* V, int64_t n, int32_t m) {
    float maxabs = 0.0f;
    for (int64_t i = 0; i < n * (int64_t)m; ++i) {
        if (!isfinite(V[i])) return NAN;
        float a = fabsf(V[i]);
        if (a > maxabs) maxabs = a;
    }
    if (maxabs == 0.0f) return 1.0f;
    float s = f32_op(FE_TONEAREST, '/', maxabs, 127.0f);
    if (s == 0.0f) s = ldexpf(1.0f, -149);
    return s;
}

/* Quantize n vectors with the given scale s: z_j = round_half_away(RN(v_j /
 * s)); returns 0, 1 for a non-finite entry, 2 for a norm bound that
 * overflows, 3 when a code would leave [-127, 127] (the vector is outside the
 * scale's range: the index rejects it rather than clip). */
int32_t orc_quantize_fixed(const float* V, int64_t n, int32_t m, int8_t* Z, int32_t ldz,
                           float s, float* s_out, float* vnorm, float* enorm, double* scratch) {
    int32_t status = 0;
    for (int64_t i = 0; i < n; ++i) {
        const float* v = V + i * (int64_t)m;
        int8_t* z = Z + i * (int64_t)ldz;
        for (int32_t j = m; j < ldz; ++j) z[j] = 0;
        int32_t st = 0;
        for (int32_t j = 0; j < m; ++j) {
            if (!isfinite(v[j])) st = 1;
        }
        if (!st) {
            for (int32_t j = 0; j < m; ++j) {
                float t = f32_op(FE_TONEAREST, '/', v[j], s);
                double r = round_half_away((double)t);
                if (r > 127.0 || r < -127.0) st = 3;
                z[j] = (int8_t)(r > 127.0 ? 127 : (r < -127.0 ? -127 : r));
            }
            for (int32_t j = 0; j < m; ++j) scratch[j] = (double)v[j];
            vnorm[i] = orc_norm_bound(scratch, m);
            for (int32_t j = 0; j < m; ++j)
                scratch[j] = (double)v[j] - (double)s * (double)z[j];
            enorm[i] = orc_norm_bound(scratch, m);
            if (!st && (isinf(vnorm[i]) || isinf(enorm[i]))) st = 2;
        }
        s_out[i] = s;
        if (st && !status) status = st;
    }
    return status;
}

/* qhat_up = norm_bound(s_q * z_q). */
float orc_qhat_norm(const int8_t* zq, float sq, int32_t m, double* scratch) {
    for (int32_t j = 0; j < m; ++j) scratch[j] = (double)sq * (double)zq[j];
    return orc_norm_bound(scratch, m);
}

/* Score interval of one corpus vector against an encoded query. */
void orc_interval_one(int64_t dot, float sq, float qnorm, float qhat, float enq,
                      float gamma, float sv, float vn, float env,
                      float* lo, float* hi) {
    float fdot = (float)dot;                     /* exact for |dot| < 2^24 */
    float ss = f32_op(FE_TONEAREST, '*', sq, sv);
    float c = f32_op(FE_TONEAREST, '*', ss, fdot);
    float e1 = f32_op(FE_UPWARD, '*', enq, vn);
    float e2 = f32_op(FE_UPWARD, '*', qhat, env);
    float E = f32_op(FE_UPWARD, '+', e1, e2);
    float g1 = f32_op(FE_UPWARD, '+', fabsf(c), E);
    float g2 = f32_op(FE_UPWARD, '*', qnorm, vn);
    float g3 = f32_op(FE_UPWARD, '+', g1, g2);
    float G = f32_op(FE_UPWARD, '*', g3, gamma);
    float r = f32_op(FE_UPWARD, '+', E, G);
    *lo = f32_op(FE_DOWNWARD, '-', c, r);
    *hi = f32_op(FE_UPWARD, '+', c, r);
}

/* Intervals of n corpus vectors (codes Z with row stride ldz) against one
 * encoded query (codes zq of length m).  The Int8 dot product is taken in
 * int64 (no overflow for any m accepted). */
void orc_intervals(const int8_t* zq, float sq, float qnorm, float qhat, float enq,
                   float gamma, const int8_t* Z, int64_t n, int32_t m, int32_t ldz,
                   const float* s, const float* vnorm, const float* enorm,
                   float* lo, float* hi) {
    for (int64_t i = 0; i < n; ++i) {
        const int8_t* zi = Z + i * (int64_t)ldz;
        int64_t dot = 0;
        for (int32_t j = 0; j < m; ++j) dot += (int64_t)zq[j] * (int64_t)zi[j];
        orc_interval_one(dot, sq, qnorm, qhat, enq, gamma, s[i], vnorm[i], enorm[i],
                         &lo[i], &hi[i]);
    }
}
