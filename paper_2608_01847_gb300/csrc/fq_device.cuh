// fq_device.cuh -- device-side building blocks of the FOCUS FP4 fake-quantizer
// (sm_103a): element / scale codecs, bf16 packing, double-fp32 arithmetic for
// the coefficient-gradient reductions, and 128-bit global accesses.
//
// Format definitions follow the paper's Sec. 3.1:
//   E2M1 elements  {0, 0.5, 1, 1.5, 2, 3, 4, 6} with sign            (Eq. 1)
//   E4M3 per-block scale of NVFP4, max 448 (E4M3FN)                   (Eq. 2)
//   E8M0 per-block scale of MXFP4, a power of two                     (Eq. 3)
// Conversions use the sm_100-family PTX cvt instructions (round to nearest
// even, saturating to the largest finite value).
#pragma once

#include <cstdint>
#include <cuda_fp16.h>
#include <cuda_runtime.h>

namespace focus {

constexpr unsigned kFullMask = 0xffffffffu;

// ---------------------------------------------------------------------------
// 32-bit division by a run-time invariant divisor (Granlund & Montgomery,
// "Division by invariant integers using multiplication", PLDI 1994, Sec. 4):
// with l = ceil(log2 d) and m = floor(2^32 (2^l - d) / d) + 1,
// n / d = (mulhi(m, n) + n) >> l for every 32-bit n.
// ---------------------------------------------------------------------------
struct FastDiv {
    uint32_t d;
    uint32_t m;
    uint32_t l;
};

inline FastDiv make_fastdiv(uint32_t d)
{
    FastDiv f;
    f.d = d;
    uint32_t l = 0;
    while ((1ull << l) < d) ++l;
    f.l = l;
    f.m = static_cast<uint32_t>((((1ull << 32) * ((1ull << l) - d)) / d) + 1);
    return f;
}

__device__ __forceinline__ uint32_t fast_div(uint32_t n, const FastDiv& f)
{
    const uint32_t t = __umulhi(n, f.m);
    return static_cast<uint32_t>((static_cast<uint64_t>(t) + n) >> f.l);
}

// ---------------------------------------------------------------------------
// bfloat16 <-> binary32
// ---------------------------------------------------------------------------
__device__ __forceinline__ float bf16_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t w) { return __uint_as_float(w & 0xffff0000u); }

// IEEE binary16 halves of a 32-bit word (exact widening) and the
// round-to-nearest-even narrowing of two floats into one word.
__device__ __forceinline__ float2 f16x2_to_float2(uint32_t w)
{
    return __half22float2(*reinterpret_cast<const __half2*>(&w));
}
__device__ __forceinline__ uint32_t pack_f16x2(float lo, float hi)
{
    const __half2 h = __floats2half2_rn(lo, hi);
    return *reinterpret_cast<const uint32_t*>(&h);
}

// Two binary32 values -> bf16x2 (round to nearest even); `lo` in bits 0-15.
__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi)
{
    uint32_t r;
    asm("cvt.rn.bf16x2.f32 %0, %1, %2;" : "=r"(r) : "f"(hi), "f"(lo));
    return r;
}

// ---------------------------------------------------------------------------
// E2M1 (Eq. 1): eight binary32 -> eight 4-bit codes in one 32-bit word,
// element 2t in the low nibble of byte t.  cvt.rn.satfinite rounds to the
// nearest E2M1 value, ties to even, and saturates at +-6; the sign is kept.
// ---------------------------------------------------------------------------
__device__ __forceinline__ uint32_t e2m1_pack8(const float (&u)[8])
{
    uint32_t r;
    asm("{\n\t.reg .b8 b0, b1, b2, b3;\n\t"
        "cvt.rn.satfinite.e2m1x2.f32 b0, %2, %1;\n\t"
        "cvt.rn.satfinite.e2m1x2.f32 b1, %4, %3;\n\t"
        "cvt.rn.satfinite.e2m1x2.f32 b2, %6, %5;\n\t"
        "cvt.rn.satfinite.e2m1x2.f32 b3, %8, %7;\n\t"
        "mov.b32 %0, {b0, b1, b2, b3};\n\t}"
        : "=r"(r)
        : "f"(u[0]), "f"(u[1]), "f"(u[2]), "f"(u[3]), "f"(u[4]), "f"(u[5]), "f"(u[6]),
          "f"(u[7]));
    return r;
}

// One byte holding two E2M1 codes -> their values as f16x2 (low nibble ->
// low half).  Exact: every E2M1 value is an f16.
__device__ __forceinline__ uint32_t e2m1x2_to_f16x2(uint32_t byte)
{
    uint32_t r;
    asm("{\n\t.reg .b8 t;\n\tcvt.u8.u32 t, %1;\n\tcvt.rn.f16x2.e2m1x2 %0, t;\n\t}"
        : "=r"(r)
        : "r"(byte));
    return r;
}

// The eight E2M1 values of a packed code word as binary32.
__device__ __forceinline__ void e2m1_unpack8(uint32_t codes, float (&q)[8])
{
#pragma unroll
    for (int b = 0; b < 4; ++b) {
        const uint32_t h2 = e2m1x2_to_f16x2((codes >> (8 * b)) & 0xffu);
        const __half2 v = *reinterpret_cast<const __half2*>(&h2);
        const float2 f = __half22float2(v);
        q[2 * b] = f.x;
        q[2 * b + 1] = f.y;
    }
}

// ---------------------------------------------------------------------------
// E4M3FN (Eq. 2): non-negative binary32 -> byte, nearest even, saturating at
// 448 (+inf -> 448); and byte -> binary32 (exact through f16).
// ---------------------------------------------------------------------------
__device__ __forceinline__ uint32_t e4m3_encode(float r)
{
    uint16_t h;
    asm("cvt.rn.satfinite.e4m3x2.f32 %0, %1, %2;" : "=h"(h) : "f"(0.0f), "f"(r));
    return h & 0xffu;
}

__device__ __forceinline__ float e4m3_decode(uint32_t byte)
{
    uint32_t r;
    asm("{\n\t.reg .b16 t;\n\tcvt.u16.u32 t, %1;\n\tcvt.rn.f16x2.e4m3x2 %0, t;\n\t}"
        : "=r"(r)
        : "r"(byte));
    return __half2float(__ushort_as_half(static_cast<unsigned short>(r & 0xffffu)));
}

// ---------------------------------------------------------------------------
// E8M0 (Eq. 3): shared exponent of an MXFP4 block with absmax m >= 0,
// clamped to [-127, 127].  rule 0 (ceiling, the paper's "typically ceiling"):
// e = ceil(log2(m / 6)), so that no |x| / 2^e exceeds 6; rule 1 (OCP MX
// v1.0): e = floor(log2 m) - 2.
// ---------------------------------------------------------------------------
__device__ __forceinline__ int mx_exponent(float m, int rule)
{
    int e;
    if (rule == 0) {
        // ceil(log2(m / 6)) of the exact quotient.  A normal binary32
        // quotient is a power of two only when m / 6 is one (m other than
        // 6 * 2^k is a relative 2^-23.6 or more away from it, fl moves by
        // 2^-24 at most); a subnormal one is not decisive (m = 0x01400001
        // rounds to 2^-127), so there m is compared with 6 * 2^-127 itself.
        const uint32_t b = __float_as_uint(__fdiv_rn(m, 6.0f));
        const int E = static_cast<int>(b >> 23);
        const uint32_t M = b & 0x7fffffu;
        e = (E == 0) ? (m > __uint_as_float(0x01400000u) ? -126 : -127)
                     : (E - 127 + (M != 0u ? 1 : 0));
    } else {
        const int E = static_cast<int>(__float_as_uint(m) >> 23);
        e = (E == 0) ? -127 : E - 129;
    }
    return min(max(e, -127), 127);
}

// ceil(log2 t) for t >= 0 clamped to [-127, 127], exact from the bits of t
// (t = 0 gives -127): the Q_E8M0 ceiling of Eq. 3 applied to a scale.
__device__ __forceinline__ int mx_ceil_exponent(float t)
{
    const uint32_t b = __float_as_uint(t);
    const int E = static_cast<int>(b >> 23);
    const uint32_t M = b & 0x7fffffu;
    const int e = (E == 0) ? (M > 0x400000u ? -126 : -127) : (E - 127 + (M != 0u ? 1 : 0));
    return min(max(e, -127), 127);
}

// 2^e for e in [-127, 127] (2^-127 is the subnormal 0x00400000).
__device__ __forceinline__ float exp2_int(int e)
{
    return (e >= -126) ? __uint_as_float(static_cast<uint32_t>(e + 127) << 23)
                       : __uint_as_float(0x00400000u);
}

// ---------------------------------------------------------------------------
// Deciding on an IEEE quotient without dividing.
//
// Several steps use a quotient q = fl(a / b) (IEEE division, round to
// nearest) only through a monotone rounding of it: its E2M1 code, the
// clipping test |q| <= 6, its E4M3 code, the E8M0 ceiling exponent.  With r
// within a few ulps of 1/b (rcp.approx.f32 is within 1 ulp), the products
//   a * fl(r * (1 - 2^-18))  and  a * fl(r * (1 + 2^-18))
// bracket q strictly (their relative distance to a/b is at least
// 2^-18 - 2^-21 > 2^-24, the most fl(a/b) can move).  A monotone rounding
// that agrees on both brackets therefore agrees on q; only when the brackets
// straddle a decision boundary is the exact quotient computed.  The estimate
// needs b and 1/b normal: exponent field of b in [2, 252].
// ---------------------------------------------------------------------------
__device__ __forceinline__ float rcp_approx(float b)
{
    float r;
    asm("rcp.approx.f32 %0, %1;" : "=f"(r) : "f"(b));
    return r;
}

constexpr float kBracketLo = 1.0f - 0x1p-18f;
constexpr float kBracketHi = 1.0f + 0x1p-18f;

__device__ __forceinline__ bool recip_ok(float b)
{
    const uint32_t E = __float_as_uint(b) >> 23;
    return (E >= 2u) && (E <= 252u);
}

struct Bracket {
    float lo, hi;  // bracketing multipliers for 1/b
    bool ok;
};

__device__ __forceinline__ Bracket make_bracket(float b)
{
    const float r = rcp_approx(b);
    return {__fmul_rn(r, kBracketLo), __fmul_rn(r, kBracketHi), recip_ok(b)};
}

// True when q' may sit within 16 encodings of a value whose encoding has its
// low LOWBITS bits clear (used for the E8M0 power-of-two test, where q' is
// within a few encodings of q).
template <int LOWBITS>
__device__ __forceinline__ bool near_threshold(float qp)
{
    constexpr uint32_t mask = (1u << LOWBITS) - 1u;
    return ((__float_as_uint(qp) + 16u) & mask) < 32u;
}

// NVFP4 block scale (Eq. 2): Delta = Q_E4M3(m / den), den = fl(alpha * 6),
// S^dq = fl(Delta * alpha); an all-zero block has Delta = 0.  `bd` brackets
// 1/den (uniform over the tensor): both brackets are converted with one
// cvt, and the exact quotient is needed only when their E4M3 codes differ.
__device__ __forceinline__ float nv_scale(float m, float alpha, float den, const Bracket& bd,
                                          uint32_t& byte)
{
    uint16_t h;
    asm("cvt.rn.satfinite.e4m3x2.f32 %0, %1, %2;"
        : "=h"(h)
        : "f"(__fmul_rn(m, bd.hi)), "f"(__fmul_rn(m, bd.lo)));
    byte = h & 0xffu;
    if (!bd.ok || (h >> 8) != byte) byte = e4m3_encode(__fdiv_rn(m, den));
    if (m == 0.0f) byte = 0u;
    return __fmul_rn(e4m3_decode(byte), alpha);
}

// MXFP4 ceiling exponent with the quotient m / 6 estimated (see above):
// only whether m / 6 is a power of two, and its binade, matter; quotients
// near the subnormal range take the exact path.
__device__ __forceinline__ int mx_exponent_fast(float m, int rule)
{
    if (rule == 0) {
        const float t = __fmul_rn(m, 1.0f / 6.0f);
        const uint32_t b = __float_as_uint(t);
        const uint32_t E = b >> 23;
        if (E >= 2u && E <= 252u && !near_threshold<23>(t))
            return min(max(static_cast<int>(E) - 126, -127), 127);  // not a power of two
    }
    return mx_exponent(m, rule);
}

// ---------------------------------------------------------------------------
// Double-fp32 ("df") arithmetic for the coefficient-gradient reductions:
// error-free transformations of Knuth (TwoSum, TAOCP vol. 2, 4.2.2),
// Dekker (Fast2Sum, Numer. Math. 18, 1971) and the FMA-based product error;
// summation is the Sum2 scheme of Ogita, Rump & Oishi (SIAM J. Sci. Comput.
// 26, 2005).  Every operation is written with an explicit rounding intrinsic
// so that no compiler contraction can change it.
// ---------------------------------------------------------------------------
struct df {
    float h, l;
};

__device__ __forceinline__ df two_sum(float a, float b)
{
    const float s = __fadd_rn(a, b);
    const float bb = __fsub_rn(s, a);
    const float e = __fadd_rn(__fsub_rn(a, __fsub_rn(s, bb)), __fsub_rn(b, bb));
    return {s, e};
}

__device__ __forceinline__ df fast_two_sum(float a, float b)
{
    const float s = __fadd_rn(a, b);
    return {s, __fsub_rn(b, __fsub_rn(s, a))};
}

__device__ __forceinline__ df df_add(df a, df b)
{
    const df s = two_sum(a.h, b.h);
    return fast_two_sum(s.h, __fadd_rn(s.l, __fadd_rn(a.l, b.l)));
}

// Add one binary32 term to a running Sum2 pair (h = sum, l = error sum).
__device__ __forceinline__ void sum2_add(df& acc, float p)
{
    const df s = two_sum(acc.h, p);
    acc.h = s.h;
    acc.l = __fadd_rn(acc.l, s.l);
}

// (a.h + a.l) / b to about 2^-44 relative, given r within a few ulps of 1/b
// (b > 0, normal): one correction step on the FMA residual.
__device__ __forceinline__ df df_div_f(df a, float b, float r)
{
    const float q1 = __fmul_rn(a.h, r);
    const float rem = __fmaf_rn(-q1, b, a.h);
    const float q2 = __fmul_rn(__fadd_rn(rem, a.l), r);
    return fast_two_sum(q1, q2);
}

__device__ __forceinline__ float df_to_f(df a) { return __fadd_rn(a.h, a.l); }

__device__ __forceinline__ df shfl_xor_df(df a, int o)
{
    return {__shfl_xor_sync(kFullMask, a.h, o), __shfl_xor_sync(kFullMask, a.l, o)};
}

// ---------------------------------------------------------------------------
// Packed binary32 pairs (sm_100-family f32x2 instructions): each lane is an
// ordinary IEEE round-to-nearest operation, two lanes per instruction.
// ---------------------------------------------------------------------------
__device__ __forceinline__ float2 mul2(float2 a, float2 b)
{
    float2 r;
    asm("{\n\t.reg .b64 ra, rb, rr;\n\t"
        "mov.b64 ra, {%2, %3};\n\tmov.b64 rb, {%4, %5};\n\t"
        "mul.rn.f32x2 rr, ra, rb;\n\tmov.b64 {%0, %1}, rr;\n\t}"
        : "=f"(r.x), "=f"(r.y)
        : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y));
    return r;
}

__device__ __forceinline__ float2 add2(float2 a, float2 b)
{
    float2 r;
    asm("{\n\t.reg .b64 ra, rb, rr;\n\t"
        "mov.b64 ra, {%2, %3};\n\tmov.b64 rb, {%4, %5};\n\t"
        "add.rn.f32x2 rr, ra, rb;\n\tmov.b64 {%0, %1}, rr;\n\t}"
        : "=f"(r.x), "=f"(r.y)
        : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y));
    return r;
}

__device__ __forceinline__ float2 sub2(float2 a, float2 b)
{
    float2 r;
    asm("{\n\t.reg .b64 ra, rb, rr;\n\t"
        "mov.b64 ra, {%2, %3};\n\tmov.b64 rb, {%4, %5};\n\t"
        "sub.rn.f32x2 rr, ra, rb;\n\tmov.b64 {%0, %1}, rr;\n\t}"
        : "=f"(r.x), "=f"(r.y)
        : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y));
    return r;
}

__device__ __forceinline__ float2 fma2(float2 a, float2 b, float2 c)
{
    float2 r;
    asm("{\n\t.reg .b64 ra, rb, rc, rr;\n\t"
        "mov.b64 ra, {%2, %3};\n\tmov.b64 rb, {%4, %5};\n\tmov.b64 rc, {%6, %7};\n\t"
        "fma.rn.f32x2 rr, ra, rb, rc;\n\tmov.b64 {%0, %1}, rr;\n\t}"
        : "=f"(r.x), "=f"(r.y)
        : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y), "f"(c.x), "f"(c.y));
    return r;
}

// Two interleaved Sum2 accumulators (even and odd terms of a sum) in one
// packed pair each: s holds the running sums, c the accumulated errors.
struct Sum2x2 {
    float2 s, c;
};

__device__ __forceinline__ void sum2x2_add(Sum2x2& a, float2 p)
{
    const float2 s = add2(a.s, p);
    const float2 bb = sub2(s, a.s);
    const float2 e = add2(sub2(a.s, sub2(s, bb)), sub2(p, bb));
    a.s = s;
    a.c = add2(a.c, e);
}

// ---------------------------------------------------------------------------
// 256-bit global accesses (sm_100 family): one 32-byte sector per lane.
// ---------------------------------------------------------------------------
__device__ __forceinline__ void ld_v8(uint32_t (&w)[8], const void* p)
{
    asm("ld.global.nc.L1::no_allocate.v8.b32 {%0, %1, %2, %3, %4, %5, %6, %7}, [%8];"
        : "=r"(w[0]), "=r"(w[1]), "=r"(w[2]), "=r"(w[3]), "=r"(w[4]), "=r"(w[5]), "=r"(w[6]),
          "=r"(w[7])
        : "l"(p));
}

__device__ __forceinline__ void st_v8(void* p, const uint32_t (&w)[8])
{
    asm volatile("st.global.cs.v8.b32 [%0], {%1, %2, %3, %4, %5, %6, %7, %8};"
                 :
                 : "l"(p), "r"(w[0]), "r"(w[1]), "r"(w[2]), "r"(w[3]), "r"(w[4]), "r"(w[5]),
                   "r"(w[6]), "r"(w[7])
                 : "memory");
}

// The same 32 bytes as two 128-bit accesses, for rows that start on a
// 16-byte but not on a 32-byte boundary.  Each of the two warp-wide loads
// touches half of every lane's sector, so the loads allocate in L1: the
// second finds the sector the first brought in.
__device__ __forceinline__ void ld_v4x2(uint32_t (&w)[8], const void* p)
{
    asm("ld.global.nc.v4.b32 {%0, %1, %2, %3}, [%8];\n\t"
        "ld.global.nc.v4.b32 {%4, %5, %6, %7}, [%8+16];"
        : "=r"(w[0]), "=r"(w[1]), "=r"(w[2]), "=r"(w[3]), "=r"(w[4]), "=r"(w[5]), "=r"(w[6]),
          "=r"(w[7])
        : "l"(p));
}

__device__ __forceinline__ void st_v4x2(void* p, const uint32_t (&w)[8])
{
    asm volatile("st.global.cs.v4.b32 [%0], {%1, %2, %3, %4};\n\t"
                 "st.global.cs.v4.b32 [%0+16], {%5, %6, %7, %8};"
                 :
                 : "l"(p), "r"(w[0]), "r"(w[1]), "r"(w[2]), "r"(w[3]), "r"(w[4]), "r"(w[5]),
                   "r"(w[6]), "r"(w[7])
                 : "memory");
}

// 32 bytes at p: one 256-bit access, or two 128-bit ones when HALF (the
// rows of the call start on 16-byte but not 32-byte boundaries; the host
// picks the kernel instantiation).
template <bool HALF>
__device__ __forceinline__ void ld_32b(uint32_t (&w)[8], const void* p)
{
    if constexpr (HALF) ld_v4x2(w, p);
    else ld_v8(w, p);
}

template <bool HALF>
__device__ __forceinline__ void st_32b(void* p, const uint32_t (&w)[8])
{
    if constexpr (HALF) st_v4x2(p, w);
    else st_v8(p, w);
}

// ---------------------------------------------------------------------------
// Global memory: one "chunk" is 8 consecutive elements of a row (16 B bf16
// or fp16, 32 B fp32), read with 128-bit non-coherent loads.
// DT: 0 binary32, 1 bfloat16, 2 binary16.
// ---------------------------------------------------------------------------
template <int DT>
struct ChunkRaw {
    uint4 w[DT != 0 ? 1 : 2];
};

template <int DT>
__device__ __forceinline__ void load_chunk(ChunkRaw<DT>& c, const void* base, uint64_t off)
{
    const uint4* p = reinterpret_cast<const uint4*>(static_cast<const char*>(base) +
                                                    off * (DT != 0 ? 2u : 4u));
    c.w[0] = __ldg(p);
    if (DT == 0) c.w[1] = __ldg(p + 1);
}

template <int DT>
__device__ __forceinline__ void zero_chunk(ChunkRaw<DT>& c)
{
    c.w[0] = make_uint4(0u, 0u, 0u, 0u);
    if (DT == 0) c.w[1] = make_uint4(0u, 0u, 0u, 0u);
}

template <int DT>
__device__ __forceinline__ void unpack_chunk(const ChunkRaw<DT>& c, float (&v)[8])
{
    if (DT == 1) {
        const uint32_t w[4] = {c.w[0].x, c.w[0].y, c.w[0].z, c.w[0].w};
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            v[2 * i] = bf16_lo(w[i]);
            v[2 * i + 1] = bf16_hi(w[i]);
        }
    } else if (DT == 2) {
        const uint32_t w[4] = {c.w[0].x, c.w[0].y, c.w[0].z, c.w[0].w};
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const float2 f = f16x2_to_float2(w[i]);
            v[2 * i] = f.x;
            v[2 * i + 1] = f.y;
        }
    } else {
#pragma unroll
        for (int i = 0; i < 2; ++i) {
            v[4 * i + 0] = __uint_as_float(c.w[i].x);
            v[4 * i + 1] = __uint_as_float(c.w[i].y);
            v[4 * i + 2] = __uint_as_float(c.w[i].z);
            v[4 * i + 3] = __uint_as_float(c.w[i].w);
        }
    }
}

template <int DT>
__device__ __forceinline__ void store_chunk(void* base, uint64_t off, const float (&v)[8])
{
    uint4* p = reinterpret_cast<uint4*>(static_cast<char*>(base) + off * (DT != 0 ? 2u : 4u));
    if (DT == 1) {
        __stcs(p, make_uint4(pack_bf16x2(v[0], v[1]), pack_bf16x2(v[2], v[3]),
                             pack_bf16x2(v[4], v[5]), pack_bf16x2(v[6], v[7])));
    } else if (DT == 2) {
        __stcs(p, make_uint4(pack_f16x2(v[0], v[1]), pack_f16x2(v[2], v[3]),
                             pack_f16x2(v[4], v[5]), pack_f16x2(v[6], v[7])));
    } else {
        __stcs(p, make_uint4(__float_as_uint(v[0]), __float_as_uint(v[1]),
                             __float_as_uint(v[2]), __float_as_uint(v[3])));
        __stcs(p + 1, make_uint4(__float_as_uint(v[4]), __float_as_uint(v[5]),
                                 __float_as_uint(v[6]), __float_as_uint(v[7])));
    }
}

}  // namespace focus
