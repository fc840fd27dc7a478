/*
 * focus_oracle.c -- CPU oracle for the FOCUS FP4 fake-quantizer
 * (Coupled-Relaxation + Dual-Granularity Scaling, MXFP4 / NVFP4).
 *
 * TEST INFRASTRUCTURE ONLY.  Only the test suite, the package smoke check and
 * the benchmark's CPU-baseline leg may load this library.  The product path
 * (the CUDA library and its Python binding) never calls it; the two share no
 * code, header, table or helper.
 *
 * This is a plain, slow, scalar restatement of the paper's definitions, one
 * block at a time, in the order the paper gives them:
 *   Sec. 3.1, Eq. 1  block fake-quantization  Xbar = Q_E2M1(X / S), Xhat = Xbar * S
 *   Sec. 3.1, Eq. 2  NVFP4 two-level scale    alpha = max|X| / (6*448),
 *                                             Delta_i = Q_E4M3(max|X_i| / (alpha*6)),
 *                                             S_i = alpha * Delta_i
 *   Sec. 3.1, Eq. 3  MXFP4 E8M0 scale         S_i = Q_E8M0(max|X_i| / 6)
 *   Sec. 3.2, Eq. 4-5 hardware scale S^dq, decoupled S^q, STE on every
 *                    non-differentiable operation
 *   Sec. 3.3, Eq. 6-7 CRS: S^q_i = S^dq_i * c_i
 *   Sec. 3.4, Eq. 8   DGS: sub-block k of block i uses S^dq_i * c_i^k
 *   Fig. 3(d)        export: only FP4 codes and dequantization scales kept
 *
 * Precision.  Every forward operation whose result is stored or decides an
 * integer (a code, a scale byte) is one IEEE-754 binary32 operation with
 * round-to-nearest-even; the library is built with -ffp-contract=off and no
 * fast-math so that no two operations are fused.  Gradient reductions are
 * accumulated in binary64 with Neumaier's compensated summation (A. Neumaier,
 * ZAMM 54, 1974) and rounded to binary32 once at the end.
 *
 * Readings of points the paper leaves open (each is listed in the design
 * notes with its justification):
 *   - E8M0 rounding: ceiling of log2 (the paper's "typically ceiling"), with
 *     the OCP MX v1.0 floor rule as an option.
 *   - E4M3 is E4M3FN (bias 7, max 448, no infinities), round-to-nearest-even
 *     with saturation to 448.
 *   - E2M1: nearest grid value, ties to the even code, saturation at 6, sign
 *     bit kept (a negative value that rounds to zero gives code 0x8, i.e. -0).
 *   - CRS and DGS combine as c_eff = fl(c_i * c_i^k); an absent coefficient
 *     array means 1.0.
 *   - STE: identity through Q_E2M1 by default (the rounding, saturation
 *     included, is the non-differentiable op); optional clipped variant that
 *     zeroes the gradient where |x / S^q| > 6.
 *   - A sub-block whose S^dq or S^q is zero or infinite is "dead": codes 0,
 *     values +0, input gradient +0, no coefficient-gradient contribution.
 *
 * Return codes: 0 ok, -1 invalid argument, -2 precondition violated
 * (non-finite input, coefficient not finite and > 0, alpha not finite >= 0).
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

enum { OR_MXFP4 = 0, OR_NVFP4 = 1 };
enum { OR_F32 = 0, OR_BF16 = 1, OR_F16 = 2 };
enum { OR_STE_IDENTITY = 0, OR_STE_CLIPPED = 1 };
enum { OR_MX_CEIL = 0, OR_MX_FLOOR = 1 };

/* ------------------------------------------------------------------ */
/* bit views                                                           */
/* ------------------------------------------------------------------ */
static float f32_of_bits(uint32_t b) { float f; memcpy(&f, &b, 4); return f; }
static uint32_t bits_of_f32(float f) { uint32_t b; memcpy(&b, &f, 4); return b; }

/* bfloat16 -> binary32 is exact: the 16 stored bits are the high half. */
static float bf16_to_f32(uint16_t h) { return f32_of_bits((uint32_t)h << 16); }

/* binary32 -> bfloat16, round to nearest, ties to even (the IEEE default
 * rounding applied to an 8-bit significand).  NaN -> canonical quiet NaN. */
uint16_t focus_oracle_bf16_rne(float f)
{
    uint32_t b = bits_of_f32(f);
    if (isnan(f)) return (uint16_t)(((b >> 16) & 0x8000u) | 0x7FC0u);
    uint32_t lsb = (b >> 16) & 1u;
    return (uint16_t)((b + 0x7FFFu + lsb) >> 16);
}

/* Round a non-negative binary64 value to the nearest integer, ties to the
 * even integer (no dependence on the floating-point environment). */
static double rne_int(double q)
{
    double f = floor(q), d = q - f;
    if (d > 0.5) return f + 1.0;
    if (d < 0.5) return f;
    return fmod(f, 2.0) != 0.0 ? f + 1.0 : f;
}

/* IEEE 754 binary16 -> binary32 (exact): sign, 5-bit exponent (bias 15),
 * 10-bit fraction; exponent 0 = subnormal m * 2^-24; 31 = inf / NaN. */
float focus_oracle_f16_decode(uint16_t h)
{
    int s = h >> 15, e = (h >> 10) & 31, m = h & 1023;
    float v;
    if (e == 0) v = ldexpf((float)m, -24);
    else if (e == 31) v = m ? NAN : INFINITY;
    else v = ldexpf((float)(1024 + m), e - 25);
    return s ? -v : v;
}

/* binary32 -> binary16, round to nearest, ties to even; magnitudes from
 * 65520 up (the midpoint above the largest finite 65504) become infinity;
 * NaN -> quiet NaN. */
uint16_t focus_oracle_f16_rne(float f)
{
    uint16_t sign = signbit(f) ? 0x8000u : 0u;
    if (isnan(f)) return (uint16_t)(sign | 0x7E00u);
    double a = fabs((double)f);
    if (a >= 65520.0) return (uint16_t)(sign | 0x7C00u);
    if (a < ldexp(1.0, -14)) {
        /* subnormal range: multiples of 2^-24 (1024 * 2^-24 is the
         * smallest normal, whose encoding 0x400 the sum below produces) */
        return (uint16_t)(sign | (uint16_t)rne_int(a * ldexp(1.0, 24)));
    }
    int ex;
    frexp(a, &ex);                          /* a in [2^(ex-1), 2^ex) */
    int E = ex - 1;
    double m = rne_int(a * ldexp(1.0, 10 - E));   /* in [1024, 2048] */
    if (m == 2048.0) { m = 1024.0; E += 1; }
    if (E + 15 >= 31) return (uint16_t)(sign | 0x7C00u);
    return (uint16_t)(sign | ((E + 15) << 10) | ((int)m - 1024));
}

/* ------------------------------------------------------------------ */
/* E2M1 element format (Eq. 1)                                         */
/* ------------------------------------------------------------------ */
/* Magnitudes by 3-bit magnitude code: the E2M1 grid {0,.5,1,1.5,2,3,4,6}. */
static const double E2M1_MAG[8] = {0.0, 0.5, 1.0, 1.5, 2.0, 3.0, 4.0, 6.0};

/* Q_E2M1 as a 4-bit code: bit 3 = sign of u, bits 0-2 = index of the nearest
 * grid magnitude; equidistant -> even index; |u| above 6 -> 6 (saturation is
 * "nearest representable value").  NaN -> code 0. */
int focus_oracle_e2m1_code(float u)
{
    if (isnan(u)) return 0;
    int sign = signbit(u) ? 8 : 0;
    double a = fabs((double)u);
    if (a >= 6.0) return sign | 7;       /* 6 is the largest value: nearest to all above */
    int best = 0;
    double bestd = fabs(a - E2M1_MAG[0]);
    for (int c = 1; c < 8; c++) {
        double d = fabs(a - E2M1_MAG[c]);
        if (d < bestd || (d == bestd && (c & 1) == 0)) { best = c; bestd = d; }
    }
    return sign | best;
}

float focus_oracle_e2m1_value(int code)
{
    float mag = (float)E2M1_MAG[code & 7];
    return (code & 8) ? -mag : mag;
}

/* ------------------------------------------------------------------ */
/* E4M3FN scale format (Eq. 2; M_FP8 = 448)                             */
/* ------------------------------------------------------------------ */
/* Decode from the bit layout: sign(1) exponent(4, bias 7) mantissa(3);
 * exponent field 0 is subnormal (m * 2^-9); 0x7F / 0xFF are NaN. */
float focus_oracle_e4m3_decode(uint8_t byte)
{
    int s = byte >> 7, e = (byte >> 3) & 15, m = byte & 7;
    if (e == 15 && m == 7) return NAN;
    double v = (e == 0) ? ldexp((double)m, -9) : ldexp(1.0 + m / 8.0, e - 7);
    return (float)(s ? -v : v);
}

/* Q_E4M3 for a non-negative ratio: nearest finite E4M3 value, ties to the
 * even code, anything at or above 448 (including +inf) -> 448 (0x7E). */
static double E4M3_TABLE[0x7F];
static int e4m3_table_ready = 0;

uint8_t focus_oracle_e4m3_encode(float r)
{
    if (!e4m3_table_ready) {             /* the decoded value of every finite code */
        for (int c = 0; c <= 0x7E; c++) E4M3_TABLE[c] = focus_oracle_e4m3_decode((uint8_t)c);
        e4m3_table_ready = 1;
    }
    if (!(r < 448.0f)) return 0x7E;     /* >= 448, +inf (NaN excluded by caller) */
    int best = 0;
    double bestd = fabs((double)r - E4M3_TABLE[0]);
    for (int c = 1; c <= 0x7E; c++) {
        double d = fabs((double)r - E4M3_TABLE[c]);
        if (d < bestd || (d == bestd && (c & 1) == 0)) { best = c; bestd = d; }
    }
    return (uint8_t)best;
}

/* ------------------------------------------------------------------ */
/* E8M0 scale format (Eq. 3)                                           */
/* ------------------------------------------------------------------ */
/* Shared exponent e of an MXFP4 block with absmax m, clamped to [-127, 127]
 * (E8M0 byte e + 127; 255 is NaN and never produced).
 *   CEIL  (default): e = ceil(log2(m / 6)) of the exact quotient (Eq. 3 with
 *                    the paper's "typically ceiling"), so |x / 2^e| <= 6.
 *                    m / 6 is evaluated in binary64: a binary32 m other
 *                    than 6 * 2^k is at least a relative 2^-23.6 away from
 *                    it (one ulp of m over 6 * 2^k), far more than binary64
 *                    rounding moves the quotient, so that quotient is a power
 *                    of two exactly when m / 6 is.  (The binary32 quotient
 *                    is not decisive: where it is subnormal, m = 0x01400001
 *                    rounds to 2^-127.)
 *   FLOOR (option):  e = floor(log2 m) - 2      -- OCP MX v1.0, 2 being the
 *                    largest E2M1 exponent. */
int focus_oracle_e8m0_exponent(float m, int rule)
{
    int e;
    if (m == 0.0f) {
        e = -127;
    } else if (rule == OR_MX_CEIL) {
        double t = (double)m / 6.0;
        int E;
        double f = frexp(t, &E);           /* t = f * 2^E, f in [0.5, 1) */
        e = (f == 0.5) ? E - 1 : E;        /* exact power of two or not */
    } else {
        int E;
        frexpf(m, &E);                     /* floor(log2 m) = E - 1 */
        e = (E - 1) - 2;
    }
    if (e < -127) e = -127;
    if (e > 127) e = 127;
    return e;
}

/* ------------------------------------------------------------------ */
/* Per-block hardware (dequantization) scale S^dq, Eq. 2-5             */
/* ------------------------------------------------------------------ */
static float block_scale(int fmt, int mx_rule, float m, float alpha, uint8_t* byte)
{
    if (fmt == OR_MXFP4) {
        int e = focus_oracle_e8m0_exponent(m, mx_rule);
        *byte = (uint8_t)(e + 127);
        return ldexpf(1.0f, e);            /* 2^-127 is a binary32 subnormal */
    }
    /* NVFP4: Delta_i = Q_E4M3(m / (alpha * 6)), S^dq = alpha * Delta_i */
    if (m == 0.0f) { *byte = 0; return 0.0f; }
    float den = alpha * 6.0f;
    float r = m / den;
    uint8_t b = focus_oracle_e4m3_encode(r);
    *byte = b;
    return focus_oracle_e4m3_decode(b) * alpha;
}

/* Hardware scale from a learnable full-precision scale S^fp (Eq. 4):
 * S^dq = Q_fmt(S^fp), the scale kept in full precision and quantized to the
 * hardware format on the fly.  MXFP4: S^fp is the block scale, rounded up to
 * a power of two (the ceiling reading of Eq. 3, so that S^fp = fl(m/6) gives
 * the absmax scale wherever fl(m/6) is a normal number).  NVFP4: alpha stays frozen and S^fp is the learnable
 * Delta^fp, S^dq = alpha * Q_E4M3(Delta^fp) (so that S^fp = fl(m/fl(alpha*6))
 * gives the absmax scale). */
static float block_scale_fp(int fmt, float sfp, float alpha, uint8_t* byte)
{
    if (fmt == OR_MXFP4) {
        int e;
        if (sfp == 0.0f) {
            e = -127;
        } else {
            int E;
            float f = frexpf(sfp, &E);
            e = (f == 0.5f) ? E - 1 : E;
        }
        if (e < -127) e = -127;
        if (e > 127) e = 127;
        *byte = (uint8_t)(e + 127);
        return ldexpf(1.0f, e);
    }
    uint8_t b = focus_oracle_e4m3_encode(sfp);
    *byte = b;
    return focus_oracle_e4m3_decode(b) * alpha;
}

/* ------------------------------------------------------------------ */
/* helpers                                                             */
/* ------------------------------------------------------------------ */
static float load_elem(int dtype, const void* p, int64_t idx)
{
    if (dtype == OR_F32) return ((const float*)p)[idx];
    if (dtype == OR_F16) return focus_oracle_f16_decode(((const uint16_t*)p)[idx]);
    return bf16_to_f32(((const uint16_t*)p)[idx]);
}

static void store_elem(int dtype, void* p, int64_t idx, float v)
{
    if (dtype == OR_F32) ((float*)p)[idx] = v;
    else if (dtype == OR_F16) ((uint16_t*)p)[idx] = focus_oracle_f16_rne(v);
    else ((uint16_t*)p)[idx] = focus_oracle_bf16_rne(v);
}

/* Neumaier-compensated binary64 running sum. */
typedef struct { double s, c; } ksum_t;
static void ksum_add(ksum_t* k, double v)
{
    double t = k->s + v;
    if (fabs(k->s) >= fabs(v)) k->c += (k->s - t) + v;
    else k->c += (v - t) + k->s;
    k->s = t;
}
static double ksum_value(const ksum_t* k) { return k->s + k->c; }

static int bad_coef(float c) { return !(isfinite(c) && c > 0.0f); }

static int check_shape(int64_t rows, int64_t cols, int64_t ld, int block, int sub, int dtype)
{
    if (rows < 0 || cols < 0 || ld < cols) return -1;
    if (block <= 0 || sub <= 0 || block % sub != 0) return -1;
    if (cols % block != 0) return -1;
    if (dtype != OR_F32 && dtype != OR_BF16 && dtype != OR_F16) return -1;
    return 0;
}

static float block_absmax(int dtype, const void* x, int64_t base, int block)
{
    float m = 0.0f;
    for (int e = 0; e < block; e++) {
        float a = fabsf(load_elem(dtype, x, base + e));
        if (a > m) m = a;
    }
    return m;
}

static int check_inputs(int fmt, int dtype, int64_t rows, int64_t cols, int64_t ld,
                        int block, int sub, int shared, const void* x,
                        const float* crs, const float* dgs, float alpha, const float* sfp)
{
    if (sfp) {
        if (shared) return -1;             /* learnable scales are per weight block */
        for (int64_t i = 0; i < rows * (cols / block); i++)
            if (!(isfinite(sfp[i]) && sfp[i] >= 0.0f)) return -2;
    }
    for (int64_t r = 0; r < rows; r++)
        for (int64_t j = 0; j < cols; j++)
            if (!isfinite(load_elem(dtype, x, r * ld + j))) return -2;
    int64_t crow = shared ? 1 : rows;
    if (crs)
        for (int64_t i = 0; i < crow * (cols / block); i++)
            if (bad_coef(crs[i])) return -2;
    if (dgs)
        for (int64_t i = 0; i < crow * (cols / sub); i++)
            if (bad_coef(dgs[i])) return -2;
    if (fmt == OR_NVFP4 && !(isfinite(alpha) && alpha >= 0.0f)) return -2;
    return 0;
}

/* ------------------------------------------------------------------ */
/* Per-tensor alpha (Eq. 2): alpha = max|X| / (M_FP4 * M_FP8) = amax / 2688 */
/* ------------------------------------------------------------------ */
int focus_oracle_alpha(int dtype, int64_t rows, int64_t cols, int64_t ld,
                       const void* x, float* alpha_out)
{
    if (rows < 0 || cols < 0 || ld < cols || !alpha_out) return -1;
    float amax = 0.0f;
    for (int64_t r = 0; r < rows; r++)
        for (int64_t j = 0; j < cols; j++) {
            float v = load_elem(dtype, x, r * ld + j);
            if (!isfinite(v)) return -2;
            float a = fabsf(v);
            if (a > amax) amax = a;
        }
    *alpha_out = amax / 2688.0f;
    return 0;
}

/* ------------------------------------------------------------------ */
/* Forward fake-quantization and export (Eq. 1-8, Fig. 3(d))            */
/* ------------------------------------------------------------------ */
/* For every block i (B contiguous elements along a row) and sub-block k
 * (sub contiguous elements of it):
 *   m       = max |x| over the block
 *   S^dq    = hardware scale (E8M0 or alpha*E4M3), scale byte
 *   c_eff   = fl(c_i * c_i^k)
 *   S^q     = fl(S^dq * c_eff)
 *   u       = fl(x / S^q),  code = Q_E2M1(u)
 *   y       = fl(value(code) * S^dq), rounded to the output dtype.
 * Outputs, each optional (NULL skips it):
 *   y      [rows, ld] in dtype (same layout as x)
 *   scales [rows, cols/block] scale bytes (E8M0 or E4M3)
 *   codes  [rows, cols/2] bytes, element 2t in the low nibble, 2t+1 high. */
int focus_oracle_fwd(int fmt, int dtype, int64_t rows, int64_t cols, int64_t ld,
                     int block, int sub, int shared, int mx_rule,
                     const void* x, const float* crs, const float* dgs, float alpha,
                     const float* sfp, void* y, uint8_t* scales, uint8_t* codes)
{
    if (check_shape(rows, cols, ld, block, sub, dtype)) return -1;
    if (fmt != OR_MXFP4 && fmt != OR_NVFP4) return -1;
    if (rows > 0 && cols > 0 && !x) return -1;
    int rc = check_inputs(fmt, dtype, rows, cols, ld, block, sub, shared, x, crs, dgs, alpha, sfp);
    if (rc) return rc;
    const int64_t nblk = cols / block, nsub = cols / sub;
    const int K = block / sub;

    for (int64_t r = 0; r < rows; r++) {
        for (int64_t j = 0; j < nblk; j++) {
            const int64_t base = r * ld + j * block;
            uint8_t sbyte;
            float s_dq = sfp ? block_scale_fp(fmt, sfp[r * nblk + j], alpha, &sbyte)
                             : block_scale(fmt, mx_rule, block_absmax(dtype, x, base, block),
                                           alpha, &sbyte);
            if (scales) scales[r * nblk + j] = sbyte;
            float c = crs ? crs[(shared ? 0 : r * nblk) + j] : 1.0f;
            for (int k = 0; k < K; k++) {
                float d = dgs ? dgs[(shared ? 0 : r * nsub) + j * K + k] : 1.0f;
                float c_eff = c * d;
                float s_q = s_dq * c_eff;
                int dead = (s_dq == 0.0f) || (s_q == 0.0f) || isinf(s_q);
                for (int e = 0; e < sub; e++) {
                    int64_t col = j * block + (int64_t)k * sub + e;
                    float xv = load_elem(dtype, x, r * ld + col);
                    int code = 0;
                    float yv = 0.0f;
                    if (!dead) {
                        float u = xv / s_q;
                        code = focus_oracle_e2m1_code(u);
                        yv = focus_oracle_e2m1_value(code) * s_dq;
                    }
                    if (y) store_elem(dtype, y, r * ld + col, yv);
                    if (codes) {
                        uint8_t* p = &codes[r * (cols / 2) + col / 2];
                        if ((col & 1) == 0) *p = (uint8_t)((*p & 0xF0) | code);
                        else *p = (uint8_t)((*p & 0x0F) | (code << 4));
                    }
                }
            }
        }
    }
    return 0;
}

/* ------------------------------------------------------------------ */
/* STE backward (Sec. 3.2: STE on all non-differentiable ops; Eq. 6-8)  */
/* ------------------------------------------------------------------ */
/* With y = Q(x / S^q) * S^dq and the STE taking dQ(u)/du = mask (1, or
 * [|u| <= 6] in the clipped variant), dy/dx = mask * S^dq / S^q:
 *   rho     = fl(S^dq / S^q)           (once per sub-block)
 *   gx      = mask ? fl(g * rho) : +0
 *   dy/dc_eff = -mask * x / c_eff^2    (S^dq cancels)
 * With T_ik = sum over sub-block (i,k) of mask*g*x and c_eff = c_i * c_i^k
 * taken exactly (binary64):
 *   dL/dc_i^k = -T_ik * c_i / c_eff^2
 *   dL/dc_i   = sum_k -T_ik * c_i^k / c_eff^2
 * In shared mode (one coefficient set for all rows) both also sum over rows.
 * With the hardware scale from a learnable S^fp (Eq. 4), the STE also gives
 *   dL/dS^dq_i = sum over block i of g * (q - mask * x / S^q)
 * (q = E2M1 value; y = q(x / S^q) * S^dq) and dL/dS^fp_i = dL/dS^dq_i for
 * MXFP4, alpha * dL/dS^dq_i for NVFP4 (STE through Q_fmt).
 * Optional outputs gcrs_abs / gdgs_abs receive the same sums taken over
 * |mask*g*x| (the scale of the terms, used to bound rounding error), and
 * gcrs64 / gdgs64 / gsfp64 the gradients themselves before the final
 * rounding to binary32 (so that partial results can be added exactly).  */
int focus_oracle_bwd(int fmt, int dtype, int64_t rows, int64_t cols, int64_t ld,
                     int block, int sub, int shared, int ste, int mx_rule,
                     const void* x, const float* crs, const float* dgs, float alpha,
                     const float* sfp, const void* g, void* gx, float* gcrs, float* gdgs,
                     float* gsfp, double* gcrs_abs, double* gdgs_abs, double* gsfp_abs,
                     double* gcrs64, double* gdgs64, double* gsfp64)
{
    if (check_shape(rows, cols, ld, block, sub, dtype)) return -1;
    if (fmt != OR_MXFP4 && fmt != OR_NVFP4) return -1;
    if (ste != OR_STE_IDENTITY && ste != OR_STE_CLIPPED) return -1;
    if (rows > 0 && cols > 0 && (!x || !g)) return -1;
    if ((gsfp || gsfp_abs || gsfp64) && shared) return -1;
    int rc = check_inputs(fmt, dtype, rows, cols, ld, block, sub, shared, x, crs, dgs, alpha, sfp);
    if (rc) return rc;
    for (int64_t r = 0; r < rows; r++)
        for (int64_t j = 0; j < cols; j++)
            if (!isfinite(load_elem(dtype, g, r * ld + j))) return -2;

    const int64_t nblk = cols / block, nsub = cols / sub;
    const int K = block / sub;

    /* shared-mode accumulators: one per coefficient, summed over all rows */
    const ksum_t zero = {0.0, 0.0};
    ksum_t* sh = 0;
    ksum_t *acc_c = 0, *acc_ca = 0, *acc_d = 0, *acc_da = 0;
    if (shared) {
        int64_t need = 2 * (nblk + nsub);
        sh = (ksum_t*)malloc((size_t)(need > 0 ? need : 1) * sizeof(ksum_t));
        if (!sh) return -1;
        for (int64_t i = 0; i < need; i++) sh[i] = zero;
        acc_c = sh; acc_ca = sh + nblk;
        acc_d = sh + 2 * nblk; acc_da = acc_d + nsub;
    }

    for (int64_t r = 0; r < rows; r++) {
        for (int64_t j = 0; j < nblk; j++) {
            const int64_t base = r * ld + j * block;
            uint8_t sbyte;
            float s_dq = sfp ? block_scale_fp(fmt, sfp[r * nblk + j], alpha, &sbyte)
                             : block_scale(fmt, mx_rule, block_absmax(dtype, x, base, block),
                                           alpha, &sbyte);
            float c = crs ? crs[(shared ? 0 : r * nblk) + j] : 1.0f;
            ksum_t gc = zero, gca = zero, gs = zero, gsa = zero;
            for (int k = 0; k < K; k++) {
                float d = dgs ? dgs[(shared ? 0 : r * nsub) + j * K + k] : 1.0f;
                float c_eff = c * d;
                float s_q = s_dq * c_eff;
                int dead = (s_dq == 0.0f) || (s_q == 0.0f) || isinf(s_q);
                /* the STE derivative of y = Q(x / S^q) * S^dq w.r.t. x is the
                 * scale ratio S^dq / S^q, rounded once for the sub-block */
                float rho = dead ? 0.0f : s_dq / s_q;
                ksum_t T = zero, Ta = zero;
                for (int e = 0; e < sub; e++) {
                    int64_t col = j * block + (int64_t)k * sub + e;
                    float xv = load_elem(dtype, x, r * ld + col);
                    float gv = load_elem(dtype, g, r * ld + col);
                    float gxv = 0.0f;
                    if (!dead) {
                        float u = xv / s_q;
                        int mask = 1;
                        if (ste == OR_STE_CLIPPED) mask = fabsf(u) <= 6.0f;
                        if (mask) {
                            gxv = gv * rho;
                            double p = (double)gv * (double)xv;   /* exact */
                            ksum_add(&T, p);
                            ksum_add(&Ta, fabs(p));
                        }
                        /* dy/dS^dq = q + S^dq * mask * du/dS^dq = q - mask * x / S^q,
                         * q from the forward's code, S^q = S^dq * c_i * c_i^k taken
                         * exactly like c_eff below */
                        double q = focus_oracle_e2m1_value(focus_oracle_e2m1_code(u));
                        double sq_exact = (double)s_dq * ((double)c * (double)d);
                        double gq = (double)gv * q;
                        double gu = mask ? (double)gv * (double)xv / sq_exact : 0.0;
                        ksum_add(&gs, gq - gu);
                        ksum_add(&gsa, fabs(gq) + fabs(gu));
                    }
                    if (gx) store_elem(dtype, gx, r * ld + col, gxv);
                }
                double ce = (double)c * (double)d;                  /* exact */
                double G = -ksum_value(&T) / (ce * ce);
                double Ga = ksum_value(&Ta) / (ce * ce);
                if (shared) {
                    ksum_add(&acc_d[j * K + k], G * (double)c);
                    ksum_add(&acc_da[j * K + k], Ga * (double)c);
                    ksum_add(&acc_c[j], G * (double)d);
                    ksum_add(&acc_ca[j], Ga * (double)d);
                } else {
                    int64_t di = r * nsub + j * K + k;
                    if (gdgs) gdgs[di] = (float)(G * (double)c);
                    if (gdgs_abs) gdgs_abs[di] = Ga * (double)c;
                    if (gdgs64) gdgs64[di] = G * (double)c;
                    ksum_add(&gc, G * (double)d);
                    ksum_add(&gca, Ga * (double)d);
                }
            }
            if (!shared) {
                if (gcrs) gcrs[r * nblk + j] = (float)ksum_value(&gc);
                if (gcrs_abs) gcrs_abs[r * nblk + j] = ksum_value(&gca);
                if (gcrs64) gcrs64[r * nblk + j] = ksum_value(&gc);
                /* STE through Q_fmt: dS^dq/dS^fp = 1 (MXFP4), alpha (NVFP4) */
                double ds = (fmt == OR_NVFP4) ? (double)alpha : 1.0;
                if (gsfp) gsfp[r * nblk + j] = (float)(ksum_value(&gs) * ds);
                if (gsfp_abs) gsfp_abs[r * nblk + j] = ksum_value(&gsa) * ds;
                if (gsfp64) gsfp64[r * nblk + j] = ksum_value(&gs) * ds;
            }
        }
    }
    if (shared) {
        for (int64_t j = 0; j < nblk; j++) {
            if (gcrs) gcrs[j] = (float)ksum_value(&acc_c[j]);
            if (gcrs_abs) gcrs_abs[j] = ksum_value(&acc_ca[j]);
            if (gcrs64) gcrs64[j] = ksum_value(&acc_c[j]);
        }
        for (int64_t i = 0; i < nsub; i++) {
            if (gdgs) gdgs[i] = (float)ksum_value(&acc_d[i]);
            if (gdgs_abs) gdgs_abs[i] = ksum_value(&acc_da[i]);
            if (gdgs64) gdgs64[i] = ksum_value(&acc_d[i]);
        }
        free(sh);
    }
    return 0;
}

/* ------------------------------------------------------------------ */
/* Dequantization of an export (the deployed-model view, Fig. 3(d))     */
/* ------------------------------------------------------------------ */
/* y = fl(value(code) * S^dq) with S^dq rebuilt from the scale byte alone:
 * 2^(byte-127) for MXFP4, fl(E4M3(byte) * alpha) for NVFP4.  y is written
 * densely as [rows, cols] in dtype. */
int focus_oracle_dequant(int fmt, int dtype, int64_t rows, int64_t cols, int block,
                         const uint8_t* codes, const uint8_t* scales, float alpha, void* y)
{
    if (rows < 0 || cols < 0 || block <= 0 || cols % block || (cols & 1)) return -1;
    if (fmt != OR_MXFP4 && fmt != OR_NVFP4) return -1;
    const int64_t nblk = cols / block;
    for (int64_t r = 0; r < rows; r++)
        for (int64_t col = 0; col < cols; col++) {
            uint8_t sb = scales[r * nblk + col / block];
            float s_dq = (fmt == OR_MXFP4) ? ldexpf(1.0f, (int)sb - 127)
                                           : focus_oracle_e4m3_decode(sb) * alpha;
            uint8_t byte = codes[r * (cols / 2) + col / 2];
            int code = (col & 1) ? (byte >> 4) : (byte & 15);
            store_elem(dtype, y, r * cols + col, focus_oracle_e2m1_value(code) * s_dq);
        }
    return 0;
}

/* ------------------------------------------------------------------ */
/* Vectorised codec entry points (used by the oracle's own pin tests)   */
/* ------------------------------------------------------------------ */
void focus_oracle_e2m1_codes(const float* u, int64_t n, uint8_t* out)
{
    for (int64_t i = 0; i < n; i++) out[i] = (uint8_t)focus_oracle_e2m1_code(u[i]);
}

void focus_oracle_e4m3_encodes(const float* r, int64_t n, uint8_t* out)
{
    for (int64_t i = 0; i < n; i++) out[i] = focus_oracle_e4m3_encode(r[i]);
}

void focus_oracle_e8m0_exponents(const float* m, int64_t n, int rule, int32_t* out)
{
    for (int64_t i = 0; i < n; i++) out[i] = focus_oracle_e8m0_exponent(m[i], rule);
}

void focus_oracle_bf16_rnes(const float* f, int64_t n, uint16_t* out)
{
    for (int64_t i = 0; i < n; i++) out[i] = focus_oracle_bf16_rne(f[i]);
}

void focus_oracle_f16_rnes(const float* f, int64_t n, uint16_t* out)
{
    for (int64_t i = 0; i < n; i++) out[i] = focus_oracle_f16_rne(f[i]);
}

void focus_oracle_f16_decodes(const uint16_t* h, int64_t n, float* out)
{
    for (int64_t i = 0; i < n; i++) out[i] = focus_oracle_f16_decode(h[i]);
}
