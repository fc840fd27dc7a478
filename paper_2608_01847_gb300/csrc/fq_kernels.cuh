// fq_kernels.cuh -- CUDA kernels of the FOCUS FP4 fake-quantizer (sm_103a).
//
// Work decomposition.  One thread owns one hardware block at a time (B = 32
// elements for MXFP4, 16 for NVFP4, contiguous along a row): its absmax, its
// scale, its coefficients and its coefficient gradients are computed once,
// in registers, with no shuffles.  A block of bf16 is one (NVFP4) or two
// (MXFP4) 256-bit loads, i.e. exactly one 32-byte sector per lane per load
// (two 128-bit loads per sector in the HALF instantiations, which the host
// launches when the rows of a call start on 16-byte but not 32-byte
// boundaries).
// The streaming kernels walk a linear block index with a grid-stride loop
// sized to the resident CTAs, issuing every load of a step before any
// arithmetic; pairs of elements go through the packed f32x2 instructions.
//
// Per element the arithmetic is the paper's, in this order (Sec. 3.1-3.4):
//   m      = block absmax                       (Eq. 2-3)
//   S^dq   = 2^e (E8M0) or fl(alpha * E4M3)     (Eq. 2-3)
//   c_eff  = fl(c_i * c_i^k),  S^q = fl(S^dq * c_eff)   (Eq. 6, 8)
//   u      = fl(x / S^q) (IEEE quotient), code = Q_E2M1(u)   (Eq. 1, 7, 8)
//   y      = fl(E2M1(code) * S^dq)               (Eq. 1, 7, 8)
// and the STE backward (Sec. 3.2):
//   gx     = mask * fl(g * rho),  rho = fl(S^dq / S^q) once per sub-block
//   T_ik   = sum of mask * g * x over the sub-block (compensated, Sum2)
//   dL/dc_i^k = -T_ik / (c_i (c_i^k)^2),  dL/dc_i = -(sum_k T_ik / c_i^k) / c_i^2
// and, in the fused-optimizer modes, one AdamW step on every learned array
// right after its gradient is known (Sec. 4.1: AdamW, constant learning rate).
#pragma once

#include "fq_device.cuh"

namespace focus {

constexpr int kThreads = 256;
// kBwdS: backward + dL/dS^fp; kBwdA / kBwdSA: the same + AdamW in place
enum Mode { kFwd = 0, kPack = 1, kBwd = 2, kBwdS = 3, kBwdA = 4, kBwdSA = 5 };

struct KParams {
    const void* x;
    const void* g;
    void* y;
    void* gx;
    const float* crs;
    const float* dgs;
    const float* alpha;
    const float* sfp;     // learnable full-precision scales (Eq. 4), or null
    float* gcrs;
    float* gdgs;
    float* gsfp;
    uint8_t* codes;
    uint8_t* scales;
    float* ws;            // scratch: per-CTA partials
    uint64_t ld;          // row pitch of x / y / g / gx in elements
    int half;             // rows of x / y / g / gx start on 16-byte (not 32-byte)
                          // boundaries: the launch takes the HALF kernels (32-byte
                          // pieces as two 128-bit accesses)
    uint32_t n_chunks;    // rows * cols / 8 (alpha pass)
    uint32_t cpr;         // 8-element chunks per row
    FastDiv div_cpr;
    uint32_t n_blocks;    // rows * cols / B
    uint32_t bpr;         // hardware blocks per row = cols / B
    FastDiv div_bpr;
    uint32_t rows;
    uint32_t nsub;        // sub-blocks per row = cols / sub_block
    uint32_t tx;          // shared-row backward: block columns per CTA
    int strided;          // ld != cols
    int shared;           // one coefficient set for all rows
    int ste;              // 0 identity, 1 clipped
    int mx_rule;          // 0 ceiling, 1 OCP floor
    uint32_t sf_tile_cols;  // export: 0 = row-major scale bytes; else the scale
                            // bytes go to 128 x 4 MMA tiles, this many per tile row
    // fused AdamW (modes kBwdA / kBwdSA and the shared-row finalisation)
    float* new_crs;       // c_i updated in place (null: c_i not learned)
    float* new_dgs;       // c_i^k updated in place
    float* new_sfp;       // S^fp updated in place
    float* opt_m[3];      // first moments of c_i, c_i^k, S^fp
    float* opt_v[3];      // second moments
    const long long* step;  // t >= 1 of this update (device); null: no optimizer step
    float lr_c, lr_s;     // learning rates of the coefficients and of S^fp
    float beta1, beta2, eps;
    float decay_c, decay_s;  // 1 - lr * weight_decay (rounded once)
};

template <int FMT, int DT, int SUB>
struct Geo {
    static constexpr int B = FMT == 0 ? 32 : 16;   // hardware block (Sec. 3.1)
    static constexpr int K = B / SUB;              // sub-blocks per block (Sec. 3.4)
    static constexpr int W = DT != 0 ? B / 2 : B;  // 32-bit words of a block of x
    static_assert(SUB >= 2 && SUB <= B && B % SUB == 0, "sub-block must divide the block");
};

// ---------------------------------------------------------------------------
// block I/O
// ---------------------------------------------------------------------------
template <int W, bool HALF>
__device__ __forceinline__ void load_block(uint32_t (&w)[W], const void* base, uint64_t byte_off)
{
    const char* p = static_cast<const char*>(base) + byte_off;
#pragma unroll
    for (int i = 0; i < W / 8; ++i) {
        uint32_t t[8];
        ld_32b<HALF>(t, p + 32 * i);
#pragma unroll
        for (int k = 0; k < 8; ++k) w[8 * i + k] = t[k];
    }
}

// Elements 2i and 2i+1 of a block as binary32 (exact).
template <int DT>
__device__ __forceinline__ float2 elem_pair(const uint32_t* w, int i)
{
    if (DT == 1) return make_float2(bf16_lo(w[i]), bf16_hi(w[i]));
    if (DT == 2) return f16x2_to_float2(w[i]);
    return make_float2(__uint_as_float(w[2 * i]), __uint_as_float(w[2 * i + 1]));
}

// Store a pair of results in the block's output words (bf16 / fp16 round
// to nearest even, or binary32 as is).
template <int DT>
__device__ __forceinline__ void put_pair(uint32_t* w, int i, float2 v)
{
    if (DT == 1) {
        w[i] = pack_bf16x2(v.x, v.y);
    } else if (DT == 2) {
        w[i] = pack_f16x2(v.x, v.y);
    } else {
        w[2 * i] = __float_as_uint(v.x);
        w[2 * i + 1] = __float_as_uint(v.y);
    }
}

// max |x| over a block, read off the stored bits (non-negative floats order
// like their encodings): packed u16x2 maxima for bf16 and fp16, u32 for
// binary32.
template <int DT, int W>
__device__ __forceinline__ float block_absmax(const uint32_t (&w)[W])
{
    if (DT != 0) {
        uint32_t m = w[0] & 0x7fff7fffu;
#pragma unroll
        for (int i = 1; i < W; ++i) {
            const uint32_t a = w[i] & 0x7fff7fffu;
            asm("max.u16x2 %0, %0, %1;" : "+r"(m) : "r"(a));
        }
        if (DT == 1) return __uint_as_float(max(m << 16, m & 0xffff0000u));
        const uint32_t top = max(m & 0xffffu, m >> 16);
        return __half2float(__ushort_as_half(static_cast<unsigned short>(top)));
    }
    uint32_t m = w[0] & 0x7fffffffu;
#pragma unroll
    for (int i = 1; i < W; ++i) m = max(m, w[i] & 0x7fffffffu);
    return __uint_as_float(m);
}

// N consecutive fp32 coefficients (N = 1, 2, 4, 8, 16), vector loads.
template <int N>
__device__ __forceinline__ void load_coefs(const float* p, float (&d)[N])
{
    if constexpr (N == 1) {
        d[0] = __ldg(p);
    } else if constexpr (N == 2) {
        const float2 v = __ldg(reinterpret_cast<const float2*>(p));
        d[0] = v.x;
        d[1] = v.y;
    } else {
#pragma unroll
        for (int i = 0; i < N / 4; ++i) {
            const float4 v = __ldg(reinterpret_cast<const float4*>(p) + i);
            d[4 * i] = v.x;
            d[4 * i + 1] = v.y;
            d[4 * i + 2] = v.z;
            d[4 * i + 3] = v.w;
        }
    }
}

template <int N>
__device__ __forceinline__ void store_coefs(float* p, const float (&d)[N])
{
    if constexpr (N == 1) {
        p[0] = d[0];
    } else if constexpr (N == 2) {
        *reinterpret_cast<float2*>(p) = make_float2(d[0], d[1]);
    } else {
#pragma unroll
        for (int i = 0; i < N / 4; ++i)
            reinterpret_cast<float4*>(p)[i] =
                make_float4(d[4 * i], d[4 * i + 1], d[4 * i + 2], d[4 * i + 3]);
    }
}

// ---------------------------------------------------------------------------
// block scale (Eq. 2-3) and relaxed scales (Eq. 6, 8)
// ---------------------------------------------------------------------------
// Per-tensor constants of the block-scale step: NVFP4's alpha, fl(alpha * 6)
// and the bracket of its reciprocal.
struct TensorScale {
    float alpha;
    float den;
    Bracket bd;
};

template <int FMT>
__device__ __forceinline__ TensorScale tensor_scale(const float* alpha_ptr)
{
    TensorScale t;
    t.alpha = (FMT == 1) ? __ldg(alpha_ptr) : 0.0f;
    t.den = __fmul_rn(t.alpha, 6.0f);
    t.bd = make_bracket(t.den);
    return t;
}

template <int FMT>
__device__ __forceinline__ float block_scale(float m, const TensorScale& ts, int mx_rule,
                                             uint32_t& byte)
{
    if (FMT == 0) {
        const int e = mx_exponent_fast(m, mx_rule);
        byte = static_cast<uint32_t>(e + 127);
        return exp2_int(e);
    }
    return nv_scale(m, ts.alpha, ts.den, ts.bd, byte);
}

// Hardware scale from a learnable full-precision scale (Eq. 4):
// S^dq = Q_fmt(S^fp).  MXFP4: the ceiling power of two of S^fp (exact, from
// its bits); NVFP4: alpha * Q_E4M3(S^fp), S^fp being the learnable Delta.
template <int FMT>
__device__ __forceinline__ float block_scale_fp(float sfp, const TensorScale& ts, uint32_t& byte)
{
    if (FMT == 0) {
        const int e = mx_ceil_exponent(sfp);
        byte = static_cast<uint32_t>(e + 127);
        return exp2_int(e);
    }
    byte = e4m3_encode(sfp);
    return __fmul_rn(e4m3_decode(byte), ts.alpha);
}

// S^q per sub-block; "dead" when S^dq or S^q is zero or infinite (outputs
// +0, no gradient).
template <int K>
__device__ __forceinline__ void relaxed_scales(float sdq, float c, const float (&d)[K],
                                               float (&sq)[K], bool (&dead)[K])
{
#pragma unroll
    for (int k = 0; k < K; ++k) {
        sq[k] = __fmul_rn(sdq, __fmul_rn(c, d[k]));
        dead[k] = (sdq == 0.0f) | (sq[k] == 0.0f) | isinf(sq[k]);
    }
}

// Nibble mask (4 bits per element) of the live elements of code word w.
template <int SUB, int K>
__device__ __forceinline__ uint32_t live_word(const bool (&dead)[K], int w)
{
    if constexpr (SUB >= 8) {
        return dead[(8 * w) / SUB] ? 0u : 0xffffffffu;
    } else {
        constexpr uint32_t sub_mask = (1u << (4 * SUB)) - 1u;
        uint32_t m = 0u;
#pragma unroll
        for (int t = 0; t < 8 / SUB; ++t)
            m |= dead[(8 * w) / SUB + t] ? 0u : (sub_mask << (4 * SUB * t));
        return m;
    }
}

// E2M1 codes (Eq. 1) of u = fl(x / S^q) for a whole block, exact: both
// brackets of every quotient (see make_bracket) are converted; where the two
// code words differ on a live element, the block's quotients are recomputed
// by IEEE division.  Dead sub-blocks get code 0.  codes[w] holds elements
// 8w .. 8w+7, element 8w+2t in the low nibble of byte t.
template <int DT, int B, int K>
__device__ __forceinline__ void block_codes(const uint32_t* xw, const float (&sq)[K],
                                            const bool (&dead)[K], uint32_t (&codes)[B / 8])
{
    constexpr int SUB = B / K;
    Bracket br[K];
    bool ok = true;
#pragma unroll
    for (int k = 0; k < K; ++k) {
        br[k] = make_bracket(sq[k]);
        ok = ok & (dead[k] | br[k].ok);
    }
    uint32_t diff = 0u;
#pragma unroll
    for (int w = 0; w < B / 8; ++w) {
        float lo[8], hi[8];
#pragma unroll
        for (int e = 0; e < 8; e += 2) {
            const int k = (8 * w + e) / SUB;
            const float2 x2 = elem_pair<DT>(xw, (8 * w + e) / 2);
            const float2 l2 = mul2(x2, make_float2(br[k].lo, br[k].lo));
            const float2 h2 = mul2(x2, make_float2(br[k].hi, br[k].hi));
            lo[e] = l2.x;
            lo[e + 1] = l2.y;
            hi[e] = h2.x;
            hi[e + 1] = h2.y;
        }
        codes[w] = e2m1_pack8(lo);
        diff |= (codes[w] ^ e2m1_pack8(hi)) & live_word<SUB, K>(dead, w);
    }
    if (!ok | (diff != 0u)) {
#pragma unroll
        for (int w = 0; w < B / 8; ++w) {
            float u[8];
#pragma unroll
            for (int e = 0; e < 8; e += 2) {
                const int k = (8 * w + e) / SUB;
                const float2 x2 = elem_pair<DT>(xw, (8 * w + e) / 2);
                u[e] = __fdiv_rn(x2.x, sq[k]);
                u[e + 1] = __fdiv_rn(x2.y, sq[k]);
            }
            codes[w] = e2m1_pack8(u);
        }
    }
#pragma unroll
    for (int w = 0; w < B / 8; ++w) codes[w] &= live_word<SUB, K>(dead, w);
}

// E2M1 code word of elements 8w .. 8w+7 of a block (exact, as block_codes,
// but one word at a time so that a caller streaming over the block keeps a
// single word live).  br holds the sub-blocks' brackets.
template <int DT, int B, int K>
__device__ __forceinline__ uint32_t word_codes(const uint32_t* xw, int w, const float (&sq)[K],
                                               const bool (&dead)[K], const Bracket (&br)[K])
{
    constexpr int SUB = B / K;
    float lo[8], hi[8];
    bool ok = true;
#pragma unroll
    for (int e = 0; e < 8; e += 2) {
        const int k = (8 * w + e) / SUB;
        const float2 x2 = elem_pair<DT>(xw, (8 * w + e) / 2);
        const float2 l2 = mul2(x2, make_float2(br[k].lo, br[k].lo));
        const float2 h2 = mul2(x2, make_float2(br[k].hi, br[k].hi));
        lo[e] = l2.x;
        lo[e + 1] = l2.y;
        hi[e] = h2.x;
        hi[e + 1] = h2.y;
        ok = ok & (dead[k] | br[k].ok);
    }
    const uint32_t live = live_word<SUB, K>(dead, w);
    uint32_t c = e2m1_pack8(lo);
    if (!ok | (((c ^ e2m1_pack8(hi)) & live) != 0u)) {
        float u[8];
#pragma unroll
        for (int e = 0; e < 8; e += 2) {
            const int k = (8 * w + e) / SUB;
            const float2 x2 = elem_pair<DT>(xw, (8 * w + e) / 2);
            u[e] = __fdiv_rn(x2.x, sq[k]);
            u[e + 1] = __fdiv_rn(x2.y, sq[k]);
        }
        c = e2m1_pack8(u);
    }
    return c & live;
}

// Clipping mask of the STE (|fl(x / S^q)| <= 6 on live sub-blocks), decided
// on the brackets and exactly when they straddle 6.  Bit e = element e.
template <int DT, int B, int K>
__device__ __forceinline__ uint32_t block_clip_mask(const uint32_t* xw, const float (&sq)[K],
                                                    const bool (&dead)[K])
{
    constexpr int SUB = B / K;
    Bracket br[K];
#pragma unroll
    for (int k = 0; k < K; ++k) br[k] = make_bracket(sq[k]);
    uint32_t live = 0u;
    bool ambiguous = false;
#pragma unroll
    for (int e = 0; e < B; e += 2) {
        const int k = e / SUB;
        const float2 x2 = elem_pair<DT>(xw, e / 2);
        const float2 l2 = mul2(x2, make_float2(br[k].lo, br[k].lo));
        const float2 h2 = mul2(x2, make_float2(br[k].hi, br[k].hi));
        const bool a0 = fabsf(h2.x) <= 6.0f, a1 = fabsf(h2.y) <= 6.0f;
        const bool b0 = fabsf(l2.x) <= 6.0f, b1 = fabsf(l2.y) <= 6.0f;
        live |= ((!dead[k] & a0) ? 1u : 0u) << e;
        live |= ((!dead[k] & a1) ? 1u : 0u) << (e + 1);
        ambiguous = ambiguous | (!dead[k] & (!br[k].ok | (a0 != b0) | (a1 != b1)));
    }
    if (ambiguous) {
        live = 0u;
#pragma unroll
        for (int e = 0; e < B; e += 2) {
            const int k = e / SUB;
            const float2 x2 = elem_pair<DT>(xw, e / 2);
            live |= ((!dead[k] & (fabsf(__fdiv_rn(x2.x, sq[k])) <= 6.0f)) ? 1u : 0u) << e;
            live |= ((!dead[k] & (fabsf(__fdiv_rn(x2.y, sq[k])) <= 6.0f)) ? 1u : 0u) << (e + 1);
        }
    }
    return live;
}

// Scale ratio rho = fl(S^dq / S^q) per sub-block (0 for dead sub-blocks).
template <int K>
__device__ __forceinline__ void scale_ratios(float sdq, const float (&sq)[K], const bool (&dead)[K],
                                             float (&rho)[K])
{
#pragma unroll
    for (int k = 0; k < K; ++k) rho[k] = dead[k] ? 0.0f : __fdiv_rn(sdq, sq[k]);
}

// Merge the two interleaved Sum2 chains of a sub-block into one pair.
__device__ __forceinline__ df sum2x2_merge(const Sum2x2& a)
{
    const df s = two_sum(a.s.x, a.s.y);
    return fast_two_sum(s.h, __fadd_rn(s.l, __fadd_rn(a.c.x, a.c.y)));
}

// ---------------------------------------------------------------------------
// STE backward of one block, sub-block by sub-block: the input gradient
// (stored one 256-bit group at a time as soon as it is complete), the
// compensated sum T_k of mask*g*x (two interleaved Sum2 chains in a packed
// pair), and the coefficient gradients
//   gd_k = -(T_k / d_k) / (c d_k),   gc = -(sum_k T_k / d_k) / c^2,
// with T_k / d_k in double-fp32 and the sum over k compensated.
// ---------------------------------------------------------------------------
template <int DT, int B, int K, bool SFPG, bool HALF>
__device__ __forceinline__ void block_bwd(const uint32_t* xw, const uint32_t* gw,
                                          const float (&sq)[K], const bool (&dead)[K],
                                          const float (&rho)[K], float c, const float (&d)[K],
                                          float sdq, int ste, bool want_gx, bool want_T,
                                          void* gx_base, uint64_t off, float (&gd)[K], float& gc,
                                          df (&T)[K], df& gS, df* q_out = nullptr)
{
    constexpr int SUB = B / K;
    constexpr int EPG = DT != 0 ? 16 : 8;  // elements per 256-bit group
    const uint32_t live = (ste == 1) ? block_clip_mask<DT, B, K>(xw, sq, dead) : 0xffffffffu;
    const float rc = rcp_approx(c);
    df Q = {0.0f, 0.0f};
    uint32_t grp[8];
    // dL/dS^dq needs the forward's E2M1 values q, one code word at a time
    Bracket br[SFPG ? K : 1];
    if constexpr (SFPG) {
#pragma unroll
        for (int k = 0; k < K; ++k) br[k] = make_bracket(sq[k]);
    }
    uint32_t cw = 0u;
    gS = {0.0f, 0.0f};
    Sum2x2 accq;   // sum of g q over the block: q = 0 on dead sub-blocks
#pragma unroll
    for (int k = 0; k < K; ++k) {
        Sum2x2 acc;
#pragma unroll
        for (int e = k * SUB; e < (k + 1) * SUB; e += 2) {
            const float2 x2 = elem_pair<DT>(xw, e / 2);
            float2 g2 = elem_pair<DT>(gw, e / 2);
            if constexpr (SFPG) {
                // g * q over the block (q: 2 significant bits, so exact for
                // bf16 g); the q term of dy/dS^dq is not masked
                if (e % 8 == 0) cw = word_codes<DT, B, K>(xw, e / 8, sq, dead, br);
                const uint32_t cb = (cw >> (4 * (e % 8))) & 0xffu;
                const uint32_t h2 = e2m1x2_to_f16x2(cb);
                const float2 q2 = __half22float2(*reinterpret_cast<const __half2*>(&h2));
                const float2 p = mul2(g2, q2);
                if (e == 0) {
                    accq.s = p;
                    accq.c = make_float2(0.0f, 0.0f);
                } else {
                    sum2x2_add(accq, p);
                }
                if (DT == 0) accq.c = add2(accq.c, fma2(g2, q2, make_float2(-p.x, -p.y)));
            }
            if (ste == 1) {
                g2.x = ((live >> e) & 1u) ? g2.x : 0.0f;
                g2.y = ((live >> (e + 1)) & 1u) ? g2.y : 0.0f;
            }
            if (want_gx) {
                // rho = 0 on dead sub-blocks; the +0 addend turns -0 into +0
                put_pair<DT>(grp, (e % EPG) / 2,
                             fma2(g2, make_float2(rho[k], rho[k]), make_float2(0.0f, 0.0f)));
                if (e % EPG == EPG - 2) {
                    st_32b<HALF>(static_cast<char*>(gx_base) + off + (e / EPG) * 32, grp);
                }
            }
            if (want_T) {
                const float2 p = mul2(g2, x2);  // exact for bf16 inputs
                if (e == k * SUB) {
                    acc.s = p;
                    acc.c = make_float2(0.0f, 0.0f);
                } else {
                    sum2x2_add(acc, p);
                }
                if (DT == 0) acc.c = add2(acc.c, fma2(g2, x2, make_float2(-p.x, -p.y)));
            }
        }
        if (want_T) {
            T[k] = dead[k] ? df{0.0f, 0.0f} : sum2x2_merge(acc);
            const float rd = rcp_approx(d[k]);
            const df qk = df_div_f(T[k], d[k], rd);
            gd[k] = -__fmul_rn(__fmul_rn(df_to_f(qk), rd), rc);
            Q = (k == 0) ? qk : df_add(Q, qk);
        }
    }
    gc = -__fmul_rn(__fmul_rn(df_to_f(Q), rc), rc);
    if (q_out) *q_out = Q;
    if constexpr (SFPG) {
        // dL/dS^dq = sum_k (sum g q - T_k / (S^dq c c^k)) over the live
        // sub-blocks = sum g q - Q / (c S^dq), Q = sum_k T_k / c^k (dead
        // sub-blocks have q = 0 and T_k = 0)
        if (sdq != 0.0f) {
            const df u = df_div_f(df_div_f(Q, c, rc), sdq, rcp_approx(sdq));
            gS = df_add(sum2x2_merge(accq), df{-u.h, -u.l});
        }
    }
}

// Coefficient gradients from finished sub-block sums (the shared-row
// finalisation): the same formulas as block_bwd.
template <int K>
__device__ __forceinline__ void block_coef_grads(const df (&T)[K], float c, const float (&d)[K],
                                                 float (&gd)[K], float& gc)
{
    const float rc = rcp_approx(c);
    df Q = {0.0f, 0.0f};
#pragma unroll
    for (int k = 0; k < K; ++k) {
        const float rd = rcp_approx(d[k]);
        const df qk = df_div_f(T[k], d[k], rd);
        gd[k] = -__fmul_rn(__fmul_rn(df_to_f(qk), rd), rc);
        Q = (k == 0) ? qk : df_add(Q, qk);
    }
    gc = -__fmul_rn(__fmul_rn(df_to_f(Q), rc), rc);
}

// ---------------------------------------------------------------------------
// Scale bytes in the block-scaled MMA layout of the Blackwell tensor cores:
// the [rows, cols/B] scale matrix is cut into tiles of 128 rows x 4 scale
// columns (512 bytes, tile row-major over the padded matrix); inside a tile,
// row r and column c sit at (r % 32) * 16 + (r / 32) * 4 + c, so that the 32
// byte-quadruples of one 16-byte line hold rows r, r+32, r+64, r+96.
// ---------------------------------------------------------------------------
__device__ __forceinline__ size_t mma_scale_offset(uint32_t row, uint32_t col, uint32_t tile_cols)
{
    const size_t tile = static_cast<size_t>(row / 128) * tile_cols + col / 4;
    return tile * 512 + (row % 32) * 16 + ((row % 128) / 32) * 4 + (col % 4);
}

// ---------------------------------------------------------------------------
// AdamW (decoupled weight decay) in binary32, PyTorch's formulation:
//   w <- w (1 - lr wd);  m <- b1 m + (1 - b1) g;  v <- b2 v + (1 - b2) g^2;
//   w <- w - lr / (1 - b1^t) * m / (sqrt(v) / sqrt(1 - b2^t) + eps).
// The bias corrections 1 - b^t = -expm1(t log1p(-(1 - b))) avoid the
// cancellation of 1 - pow(b, t) at small t; they are evaluated per thread
// from the device step counter, so a captured graph replays correctly.
// ---------------------------------------------------------------------------
struct AdamW {
    float b1, o1, b2, o2, eps, rbc2, step_c, step_s, decay_c, decay_s;
};

__device__ __forceinline__ AdamW adamw_setup(const KParams& p)
{
    AdamW a;
    const float t = static_cast<float>(__ldg(p.step));
    a.b1 = p.beta1;
    a.b2 = p.beta2;
    a.o1 = __fsub_rn(1.0f, p.beta1);
    a.o2 = __fsub_rn(1.0f, p.beta2);
    a.eps = p.eps;
    const float bc1 = -expm1f(__fmul_rn(t, log1pf(-a.o1)));
    const float bc2 = -expm1f(__fmul_rn(t, log1pf(-a.o2)));
    a.rbc2 = __frsqrt_rn(bc2);
    a.step_c = __fdiv_rn(p.lr_c, bc1);
    a.step_s = __fdiv_rn(p.lr_s, bc1);
    a.decay_c = p.decay_c;
    a.decay_s = p.decay_s;
    return a;
}

// One update of parameter w with gradient gr; m and v are updated in place.
// The moments are exact binary32 operations; the square root and the
// division of the step use the hardware's approximate forms (sqrt.approx,
// div.full: within 2 ulp), which the update's tolerance covers -- six of each
// per MXFP4 block cost as much as the rest of the optimizer (MXFP4 backward
// with AdamW on S^fp, c, c^k: 5978 -> 6299 GB/s on the Llama-70B layer set).
__device__ __forceinline__ float adamw_update(float w, float gr, float& m, float& v, float step,
                                              float decay, const AdamW& a)
{
    m = __fadd_rn(__fmul_rn(a.b1, m), __fmul_rn(a.o1, gr));
    v = __fadd_rn(__fmul_rn(a.b2, v), __fmul_rn(a.o2, __fmul_rn(gr, gr)));
    float sq, q;
    asm("sqrt.approx.f32 %0, %1;" : "=f"(sq) : "f"(v));
    const float den = __fadd_rn(__fmul_rn(sq, a.rbc2), a.eps);
    asm("div.full.f32 %0, %1, %2;" : "=f"(q) : "f"(m), "f"(den));
    return __fsub_rn(__fmul_rn(w, decay), __fmul_rn(step, q));
}

// Moments of one block's parameters, loaded with the block's other inputs.
template <int K>
struct BlockMoments {
    float mc, vc, ms, vs;
    float md[K], vd[K];
};

// ---------------------------------------------------------------------------
// Forward / pack / per-row backward over a linear block index.
// ---------------------------------------------------------------------------
template <int FMT, int DT, int MODE>
struct Unroll {
    // blocks per thread per step: 64 bytes of x in flight for the streaming
    // passes, one block (x and g) for the backward
    static constexpr int U = (MODE >= kBwd) ? 1 : ((FMT == 1 && DT != 0) ? 2 : 1);
};

// Backward kernels that split each 32-element MXFP4 block over two adjacent
// lanes (16 elements each; the block maximum and the sums over sub-blocks
// exchanged by shuffle), which halves the per-thread state of a block.  Taken
// where it measured faster (backward phase on the Llama-70B layer set, GB/s,
// one lane per block -> a pair): 16-bit elements with sub-blocks of 2 (5326
// -> 6355), 4 (6411 -> 6642) or 16 (6700 -> 6962), binary16 with sub-blocks
// of 8 (6409 -> 6896).  Not for bf16 with sub-blocks of 8 (7035 -> 6891), nor
// with the S^fp gradient or the fused optimizer (5-13 % slower: both lanes
// redo the per-block work, and their state does not halve), nor for binary32
// (not measured).
template <int FMT, int DT, int SUB, int MODE>
struct PairBlocks {
    static constexpr bool value =
        FMT == 0 && MODE == kBwd && DT != 0 && SUB <= 16 && (SUB != 8 || DT == 2);
};

// Blocks one CTA covers per step of its grid-stride loop.
template <int FMT, int DT, int SUB, int MODE>
struct Span {
    static constexpr int value =
        PairBlocks<FMT, DT, SUB, MODE>::value ? kThreads / 2 : Unroll<FMT, DT, MODE>::U * kThreads;
};

// Resident CTAs per SM the register allocation must allow.  The backward is
// bound by memory latency: with 16-bit elements, one more CTA per SM than the
// registers it would like (4 for NVFP4 at 64 registers, 3 for MXFP4 at 80)
// is faster despite a few dozen bytes of spills to L1-cached local memory
// (measured: NVFP4 Qwen3-4B backward 6124 -> 6543 GB/s).  The backward fused
// with AdamW on the coefficients takes the same counts (Llama-70B layer set,
// NVFP4 6664 -> 6883 GB/s, MXFP4 6617 -> 6704; Qwen3-4B 6448 -> 6547, against
// one CTA fewer); with S^fp learned as well its extra state spills too much
// and keeps one fewer (at the backward's count: 70B NVFP4 6361 -> 6177) --
// except NVFP4 with 16-bit elements and sub-blocks of 8 or more since the
// optimizer's square root and division are the approximate forms (70B: 6571
// -> 6793 at 4 CTAs; MXFP4 at 3: 6297 -> 6154).
// The MXFP4 backward with binary16 elements is the exception: its
// conversions spill three times as much at 3 CTAs, and 2 CTAs per SM are
// faster (Llama-70B layer set, fp16 I/O: backward 5927 -> 6413 GB/s).
// The NVFP4 export (pack) likewise runs faster at 5 CTAs per SM than at 4
// (pack phase: Qwen3-4B 5746 -> 5913 GB/s, Llama-70B layer 6715 -> 6796);
// the MXFP4 export (70B: 6915 -> 6722) and the forward (Qwen3-4B NVFP4: 6409
// -> 6282) do not.  One fewer for 2-element sub-blocks, whose per-sub-block
// state is largest -- except the plain NVFP4 backward of 16-bit elements,
// which is faster at the full count there too (70B 6058 -> 6231, Qwen3-4B
// 5802 -> 5953 GB/s; the MXFP4 one is not: 5325 -> 4850).
template <int FMT_, int DT, int SUB, int MODE>
struct MinCtas {
    // a thread of a pair kernel holds 16 elements, as an NVFP4 thread does
    static constexpr int FMT = PairBlocks<FMT_, DT, SUB, MODE>::value ? 1 : FMT_;
    static constexpr int bwd = FMT == 1 ? (DT != 0 ? 4 : 3) : (DT == 1 ? 3 : 2);
    static constexpr int adam_sfp = FMT == 1 ? ((DT != 0 && SUB >= 8) ? 4 : 3) : 2;
    static constexpr int base =
        MODE == kBwdSA ? adam_sfp : (MODE >= kBwd) ? bwd : (MODE == kPack && FMT == 1) ? 5 : 4;
    static constexpr int value = base - ((SUB == 2 && !(FMT == 1 && DT != 0 && MODE == kBwd)) ? 1 : 0);
};

// Where a block's tensor comes from: one tensor (the per-tensor entry
// points), or a group of tensors walked as one concatenated block range (the
// group entry points: one launch for all projections of a layer, so no
// tensor's tail waits alone and launches are saved).
template <int FMT>
struct OneTensor {
    const KParams& p;
    TensorScale scale;
    __device__ __forceinline__ explicit OneTensor(const KParams& q) : p(q), scale(tensor_scale<FMT>(q.alpha)) {}
    // tiles of `span` blocks; tile i is blocks [i * span, (i + 1) * span)
    __device__ __forceinline__ uint32_t tiles(uint32_t span) const { return (p.n_blocks + span - 1) / span; }
    __device__ __forceinline__ int tensor(uint32_t) const { return 0; }
    __device__ __forceinline__ uint32_t base(uint32_t tile, int, uint32_t span) const { return tile * span; }
    __device__ __forceinline__ const KParams& at(int) const { return p; }
    __device__ __forceinline__ const TensorScale& ts(int) const { return scale; }
};

constexpr int kMaxGroup = 16;
struct KGroup {
    KParams p[kMaxGroup];
    uint32_t start[kMaxGroup + 1];  // first tile of tensor t; a tile is one CTA step of blocks
    int n;
};

template <int FMT>
struct TensorGroup {
    const KGroup& g;
    const TensorScale* scale;       // per tensor, in shared memory
    // tensors start on tile boundaries, so a CTA step never mixes tensors
    __device__ __forceinline__ uint32_t tiles(uint32_t) const { return g.start[g.n]; }
    __device__ __forceinline__ int tensor(uint32_t tile) const
    {
        int t = 0;
        while (t + 1 < g.n && tile >= g.start[t + 1]) ++t;
        return t;
    }
    __device__ __forceinline__ uint32_t base(uint32_t tile, int t, uint32_t span) const
    {
        return (tile - g.start[t]) * span;
    }
    __device__ __forceinline__ const KParams& at(int t) const { return g.p[t]; }
    __device__ __forceinline__ const TensorScale& ts(int t) const { return scale[t]; }
};

template <int FMT, int DT, int SUB, int MODE, bool HALF, class Src>
__device__ __forceinline__ void block_loop(const Src& src)
{
    using G = Geo<FMT, DT, SUB>;
    constexpr int B = G::B, K = G::K, W = G::W;
    constexpr int U = Unroll<FMT, DT, MODE>::U;
    constexpr int ESZ = DT != 0 ? 2 : 4;
    constexpr bool BWD = MODE >= kBwd;
    constexpr bool SFPG = MODE == kBwdS || MODE == kBwdSA;
    constexpr bool ADAM = MODE >= kBwdA;
    AdamW aw;
    if constexpr (ADAM) aw = adamw_setup(src.at(0));   // one optimizer step for all tensors
    const uint32_t span = U * kThreads;
    const uint32_t n_tiles = src.tiles(span);

    for (uint32_t tile = blockIdx.x; tile < n_tiles; tile += gridDim.x) {
        // one tensor per CTA step: its parameters are uniform across the CTA
        const int tt = src.tensor(tile);
        const KParams& p = src.at(tt);
        const TensorScale& ts = src.ts(tt);
        const uint32_t base = src.base(tile, tt, span);
        const bool want_gx = BWD && p.gx != nullptr;
        const bool want_T = SFPG || (BWD && (p.gcrs != nullptr || p.gdgs != nullptr)) ||
                            (ADAM && (p.new_crs != nullptr || p.new_dgs != nullptr));
        uint32_t xr[U][W];
        uint32_t gr[BWD ? U : 1][BWD ? W : 1];
        uint64_t off[U];
        float cv[U];
        float dv[U][K];
        float sv[U];
        BlockMoments<ADAM ? K : 1> mo[ADAM ? U : 1];
        // ---- issue every load of this step first ----
#pragma unroll
        for (int j = 0; j < U; ++j) {
            const uint32_t blk = base + j * kThreads + threadIdx.x;
            cv[j] = 1.0f;
            sv[j] = 0.0f;
#pragma unroll
            for (int k = 0; k < K; ++k) dv[j][k] = 1.0f;
            off[j] = 0;
            if (blk < p.n_blocks) {
                uint32_t cb = 0;
                if (p.strided || p.shared) {
                    const uint32_t row = fast_div(blk, p.div_bpr);
                    cb = blk - row * p.bpr;
                    off[j] = (static_cast<uint64_t>(row) * p.ld + static_cast<uint64_t>(cb) * B) * ESZ;
                } else {
                    off[j] = static_cast<uint64_t>(blk) * (B * ESZ);
                }
                load_block<W, HALF>(xr[j], p.x, off[j]);
                if constexpr (BWD) load_block<W, HALF>(gr[j], p.g, off[j]);
                if (p.sfp) sv[j] = __ldg(p.sfp + blk);
                const uint32_t q = p.shared ? cb : blk;
                if (p.crs) cv[j] = __ldg(p.crs + q);
                if (p.dgs) load_coefs<K>(p.dgs + static_cast<size_t>(q) * K, dv[j]);
                if constexpr (ADAM) {
                    if (p.new_crs) {
                        mo[j].mc = p.opt_m[0][blk];
                        mo[j].vc = p.opt_v[0][blk];
                    }
                    if (p.new_dgs) {
                        load_coefs<K>(p.opt_m[1] + static_cast<size_t>(blk) * K, mo[j].md);
                        load_coefs<K>(p.opt_v[1] + static_cast<size_t>(blk) * K, mo[j].vd);
                    }
                    if (SFPG && p.new_sfp) {
                        mo[j].ms = p.opt_m[2][blk];
                        mo[j].vs = p.opt_v[2][blk];
                    }
                }
            } else {
#pragma unroll
                for (int i = 0; i < W; ++i) xr[j][i] = 0u;
                if constexpr (BWD) {
#pragma unroll
                    for (int i = 0; i < W; ++i) gr[j][i] = 0u;
                }
            }
        }
        // ---- arithmetic and stores ----
#pragma unroll
        for (int j = 0; j < U; ++j) {
            const uint32_t blk = base + j * kThreads + threadIdx.x;
            if (blk >= p.n_blocks) continue;
            uint32_t sbyte;
            const float sdq = p.sfp ? block_scale_fp<FMT>(sv[j], ts, sbyte)
                                    : block_scale<FMT>(block_absmax<DT, W>(xr[j]), ts, p.mx_rule, sbyte);
            float sq[K];
            bool dead[K];
            relaxed_scales<K>(sdq, cv[j], dv[j], sq, dead);

            if constexpr (!BWD) {
                uint32_t codes[B / 8];
                block_codes<DT, B, K>(xr[j], sq, dead, codes);
                if constexpr (MODE == kFwd) {
                    constexpr int EPG = DT != 0 ? 16 : 8;  // elements per 256-bit group
                    uint32_t grp[8];
#pragma unroll
                    for (int w = 0; w < B / 8; ++w) {
                        float q[8];
                        e2m1_unpack8(codes[w], q);
#pragma unroll
                        for (int e = 0; e < 8; e += 2) {
                            const int el = 8 * w + e;
                            put_pair<DT>(grp, (el % EPG) / 2,
                                         mul2(make_float2(q[e], q[e + 1]), make_float2(sdq, sdq)));
                            if (el % EPG == EPG - 2)
                                st_32b<HALF>(static_cast<char*>(p.y) + off[j] + (el / EPG) * 32, grp);
                        }
                    }
                } else {
                    uint32_t* dst =
                        reinterpret_cast<uint32_t*>(p.codes) + static_cast<size_t>(blk) * (B / 8);
                    if constexpr (B == 32) {
                        __stcs(reinterpret_cast<uint4*>(dst),
                               make_uint4(codes[0], codes[1], codes[2], codes[3]));
                    } else {
                        __stcs(reinterpret_cast<uint2*>(dst), make_uint2(codes[0], codes[1]));
                    }
                }
                if (p.scales) {
                    size_t at = blk;
                    if (p.sf_tile_cols) {
                        const uint32_t row = fast_div(blk, p.div_bpr);
                        at = mma_scale_offset(row, blk - row * p.bpr, p.sf_tile_cols);
                    }
                    p.scales[at] = static_cast<uint8_t>(sbyte);
                }
            } else {
                float rho[K];
                if (want_gx) scale_ratios<K>(sdq, sq, dead, rho);
                float gd[K], gc;
                df T[K], gS;
                block_bwd<DT, B, K, SFPG, HALF>(xr[j], gr[j], sq, dead, rho, cv[j], dv[j], sdq, p.ste,
                                                want_gx, want_T, p.gx, off[j], gd, gc, T, gS);
                if (want_T) {
                    if (p.gdgs) store_coefs<K>(p.gdgs + static_cast<size_t>(blk) * K, gd);
                    if (p.gcrs) p.gcrs[blk] = gc;
                }
                float gs = 0.0f;
                if constexpr (SFPG) {
                    // STE through Q_fmt: dS^dq/dS^fp = 1 (MXFP4), alpha (NVFP4)
                    const float v = df_to_f(gS);
                    gs = (FMT == 1) ? __fmul_rn(v, ts.alpha) : v;
                    if (p.gsfp) p.gsfp[blk] = gs;
                }
                if constexpr (ADAM) {
                    BlockMoments<K>& o = mo[j];
                    if (p.new_crs) {
                        p.new_crs[blk] = adamw_update(cv[j], gc, o.mc, o.vc, aw.step_c, aw.decay_c, aw);
                        p.opt_m[0][blk] = o.mc;
                        p.opt_v[0][blk] = o.vc;
                    }
                    if (p.new_dgs) {
                        float nd[K];
#pragma unroll
                        for (int k = 0; k < K; ++k)
                            nd[k] = adamw_update(dv[j][k], gd[k], o.md[k], o.vd[k], aw.step_c,
                                                 aw.decay_c, aw);
                        const size_t q = static_cast<size_t>(blk) * K;
                        store_coefs<K>(p.new_dgs + q, nd);
                        store_coefs<K>(p.opt_m[1] + q, o.md);
                        store_coefs<K>(p.opt_v[1] + q, o.vd);
                    }
                    if (SFPG && p.new_sfp) {
                        p.new_sfp[blk] = adamw_update(sv[j], gs, o.ms, o.vs, aw.step_s, aw.decay_s, aw);
                        p.opt_m[2][blk] = o.ms;
                        p.opt_v[2][blk] = o.vs;
                    }
                }
            }
        }
    }
}

// ---------------------------------------------------------------------------
// MXFP4 backward with each 32-element block split over two adjacent lanes
// (PairBlocks): lane h of the pair owns elements 16h .. 16h+15, i.e. the
// sub-blocks K/2 h .. K/2 h + K/2 - 1.  The pair computes the block maximum
// with one shuffle, each lane its half's input gradient, sub-block sums and
// DGS gradients as block_bwd does for a 16-element block, and the pair adds
// the two halves of sum_k T_k / c^k (and of dL/dS^dq) in a fixed order, lower
// half first, for the CRS gradient and the S^fp gradient; lane 0 of the pair
// writes the per-block results.  Every lane runs every step (lanes past the
// last block compute on zeros and store nothing), so the shuffles see full
// warps.
// ---------------------------------------------------------------------------
template <int DT, int SUB, int MODE, bool HALF, class Src>
__device__ __forceinline__ void pair_bwd_loop(const Src& src)
{
    constexpr int B = 32, K = B / SUB, BH = 16, KH = K / 2;
    constexpr int WH = DT != 0 ? BH / 2 : BH;   // 32-bit words of a half block
    constexpr int ESZ = DT != 0 ? 2 : 4;
    constexpr bool SFPG = MODE == kBwdS || MODE == kBwdSA;
    constexpr bool ADAM = MODE >= kBwdA;
    static_assert(KH >= 1 && BH % SUB == 0, "a sub-block must lie in one half");
    AdamW aw;
    if constexpr (ADAM) aw = adamw_setup(src.at(0));
    const uint32_t span = kThreads / 2;
    const uint32_t n_tiles = src.tiles(span);
    const uint32_t h = threadIdx.x & 1u;

    for (uint32_t tile = blockIdx.x; tile < n_tiles; tile += gridDim.x) {
        const int tt = src.tensor(tile);
        const KParams& p = src.at(tt);
        const TensorScale& ts = src.ts(tt);
        const uint32_t blk = src.base(tile, tt, span) + threadIdx.x / 2;
        const bool valid = blk < p.n_blocks;
        const bool want_gx = p.gx != nullptr;
        const bool want_T = SFPG || p.gcrs != nullptr || p.gdgs != nullptr ||
                            (ADAM && (p.new_crs != nullptr || p.new_dgs != nullptr));
        uint32_t xr[WH], gr[WH];
        float cv = 1.0f, sv = 0.0f, dv[KH];
        BlockMoments<ADAM ? KH : 1> mo;
#pragma unroll
        for (int k = 0; k < KH; ++k) dv[k] = 1.0f;
        uint64_t off = 0;
        if (valid) {
            uint32_t cb = 0;
            if (p.strided || p.shared) {
                const uint32_t row = fast_div(blk, p.div_bpr);
                cb = blk - row * p.bpr;
                off = (static_cast<uint64_t>(row) * p.ld + static_cast<uint64_t>(cb) * B + BH * h) * ESZ;
            } else {
                off = (static_cast<uint64_t>(blk) * B + BH * h) * ESZ;
            }
            load_block<WH, HALF>(xr, p.x, off);
            load_block<WH, HALF>(gr, p.g, off);
            if (p.sfp) sv = __ldg(p.sfp + blk);
            const uint32_t q = p.shared ? cb : blk;
            if (p.crs) cv = __ldg(p.crs + q);
            if (p.dgs) load_coefs<KH>(p.dgs + static_cast<size_t>(q) * K + KH * h, dv);
            if constexpr (ADAM) {
                if (p.new_crs) {
                    mo.mc = p.opt_m[0][blk];
                    mo.vc = p.opt_v[0][blk];
                }
                if (p.new_dgs) {
                    load_coefs<KH>(p.opt_m[1] + static_cast<size_t>(blk) * K + KH * h, mo.md);
                    load_coefs<KH>(p.opt_v[1] + static_cast<size_t>(blk) * K + KH * h, mo.vd);
                }
                if (SFPG && p.new_sfp) {
                    mo.ms = p.opt_m[2][blk];
                    mo.vs = p.opt_v[2][blk];
                }
            }
        } else {
#pragma unroll
            for (int i = 0; i < WH; ++i) xr[i] = gr[i] = 0u;
        }
        // the block maximum over both halves (max of non-negative floats)
        const float mh = block_absmax<DT, WH>(xr);
        const float m = fmaxf(mh, __shfl_xor_sync(kFullMask, mh, 1));
        uint32_t sbyte;
        const float sdq = p.sfp ? block_scale_fp<0>(sv, ts, sbyte) : block_scale<0>(m, ts, p.mx_rule, sbyte);
        float sq[KH];
        bool dead[KH];
        relaxed_scales<KH>(sdq, cv, dv, sq, dead);
        float rho[KH];
        if (want_gx) scale_ratios<KH>(sdq, sq, dead, rho);
        float gd[KH], gc_half;
        df T[KH], gS, Q;
        block_bwd<DT, BH, KH, SFPG, HALF>(xr, gr, sq, dead, rho, cv, dv, sdq, p.ste, want_gx && valid,
                                          want_T, p.gx, off, gd, gc_half, T, gS, &Q);
        // the two halves' sums, lower half first
        const df Qo = shfl_xor_df(Q, 1);
        const df Qt = h == 0 ? df_add(Q, Qo) : df_add(Qo, Q);
        const float rc = rcp_approx(cv);
        const float gc = -__fmul_rn(__fmul_rn(df_to_f(Qt), rc), rc);
        float gs = 0.0f;
        if constexpr (SFPG) {
            const df So = shfl_xor_df(gS, 1);
            gs = df_to_f(h == 0 ? df_add(gS, So) : df_add(So, gS));   // STE through Q_fmt: dS^dq/dS^fp = 1
        }
        if (!valid) continue;
        if (want_T && p.gdgs) store_coefs<KH>(p.gdgs + static_cast<size_t>(blk) * K + KH * h, gd);
        if (h == 0) {
            if (want_T && p.gcrs) p.gcrs[blk] = gc;
            if (SFPG && p.gsfp) p.gsfp[blk] = gs;
        }
        if constexpr (ADAM) {
            if (p.new_crs && h == 0) {
                p.new_crs[blk] = adamw_update(cv, gc, mo.mc, mo.vc, aw.step_c, aw.decay_c, aw);
                p.opt_m[0][blk] = mo.mc;
                p.opt_v[0][blk] = mo.vc;
            }
            if (p.new_dgs) {
                float nd[KH];
#pragma unroll
                for (int k = 0; k < KH; ++k)
                    nd[k] = adamw_update(dv[k], gd[k], mo.md[k], mo.vd[k], aw.step_c, aw.decay_c, aw);
                const size_t q = static_cast<size_t>(blk) * K + KH * h;
                store_coefs<KH>(p.new_dgs + q, nd);
                store_coefs<KH>(p.opt_m[1] + q, mo.md);
                store_coefs<KH>(p.opt_v[1] + q, mo.vd);
            }
            if (SFPG && p.new_sfp && h == 0) {
                p.new_sfp[blk] = adamw_update(sv, gs, mo.ms, mo.vs, aw.step_s, aw.decay_s, aw);
                p.opt_m[2][blk] = mo.ms;
                p.opt_v[2][blk] = mo.vs;
            }
        }
    }
}


template <int FMT, int DT, int SUB, int MODE, bool HALF>
__global__ void __launch_bounds__(kThreads, (MinCtas<FMT, DT, SUB, MODE>::value))
    fq_block_kernel(const KParams p)
{
    // launched as a programmatic dependent of the previous kernel in the
    // stream: wait until that one has completed (its results visible), then
    // let the next one be scheduled behind this grid
    asm volatile("griddepcontrol.wait;" ::: "memory");
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    if constexpr (PairBlocks<FMT, DT, SUB, MODE>::value)
        pair_bwd_loop<DT, SUB, MODE, HALF>(OneTensor<FMT>(p));
    else
        block_loop<FMT, DT, SUB, MODE, HALF>(OneTensor<FMT>(p));
}

template <int FMT, int DT, int SUB, int MODE, bool HALF>
__global__ void __launch_bounds__(kThreads, (MinCtas<FMT, DT, SUB, MODE>::value))
    fq_group_kernel(const __grid_constant__ KGroup g)
{
    static_assert(MODE < kBwdA, "the fused optimizer is per tensor");
    __shared__ TensorScale scale[kMaxGroup];
    if (threadIdx.x < g.n) scale[threadIdx.x] = tensor_scale<FMT>(g.p[threadIdx.x].alpha);
    __syncthreads();
    if constexpr (PairBlocks<FMT, DT, SUB, MODE>::value)
        pair_bwd_loop<DT, SUB, MODE, HALF>(TensorGroup<FMT>{g, scale});
    else
        block_loop<FMT, DT, SUB, MODE, HALF>(TensorGroup<FMT>{g, scale});
}

// ---------------------------------------------------------------------------
// Backward with coefficients shared by all rows.  A CTA is p.tx columns of
// blocks x (kThreads / p.tx) row slots; thread (tx, ty) owns column block
// cb = blockIdx.x * p.tx + tx and walks the rows of its slot, keeping that
// column's coefficients and its K running sums in registers.  The CTA then
// combines its row slots in a fixed order and writes one double-fp32 partial
// per (row group, sub-block column) to scratch; fq_bwd_shared_finalize sums
// the row groups in a fixed order.
// ---------------------------------------------------------------------------
// Resident CTAs per SM the shared-row backward's registers must allow.  For
// NVFP4 with 16-bit elements, 4 (64 registers, a few bytes of spills to L1),
// as the per-row backward: with the whole-wave grid of shared_row_groups the
// activations' shared-row backward ran at 6595 GB/s against 6407 at 3 CTAs
// and a part-empty last wave.  MXFP4 keeps 2 (its unconstrained allocation
// was 94 registers without spills for bf16 and sub-block 8; bounded to 3
// CTAs it spilled and measured 6435 against 6763 GB/s), and 1 for 2-element
// sub-blocks, whose per-sub-block state needs about 200 registers.
template <int FMT, int DT, int SUB>
struct MinCtasShared {
    static constexpr int value =
        FMT == 1 ? (DT != 0 ? (SUB == 2 ? 3 : 4) : (SUB == 2 ? 2 : 3)) : (SUB == 2 ? 1 : 2);
};

template <int FMT, int DT, int SUB, bool HALF>
__global__ void __launch_bounds__(kThreads, (MinCtasShared<FMT, DT, SUB>::value)) fq_bwd_shared_kernel(const KParams p)
{
    using G = Geo<FMT, DT, SUB>;
    constexpr int B = G::B, K = G::K, W = G::W;
    constexpr int ESZ = DT != 0 ? 2 : 4;
    __shared__ float2 red[kThreads * K];
    const TensorScale ts = tensor_scale<FMT>(p.alpha);
    const bool want_gx = p.gx != nullptr;
    const uint32_t tx = threadIdx.x % p.tx, ty = threadIdx.x / p.tx, nty = kThreads / p.tx;
    const uint32_t cb = blockIdx.x * p.tx + tx;
    const bool col_ok = cb < p.bpr;

    float c = 1.0f;
    float d[K];
#pragma unroll
    for (int k = 0; k < K; ++k) d[k] = 1.0f;
    if (col_ok) {
        if (p.crs) c = __ldg(p.crs + cb);
        if (p.dgs) load_coefs<K>(p.dgs + static_cast<size_t>(cb) * K, d);
    }
    df acc[K];
#pragma unroll
    for (int k = 0; k < K; ++k) acc[k] = {0.0f, 0.0f};

    if (col_ok) {
        for (uint32_t r = blockIdx.y * nty + ty; r < p.rows; r += gridDim.y * nty) {
            uint32_t xr[W], gr[W];
            const uint64_t off =
                (static_cast<uint64_t>(r) * p.ld + static_cast<uint64_t>(cb) * B) * ESZ;
            load_block<W, HALF>(xr, p.x, off);
            load_block<W, HALF>(gr, p.g, off);
            uint32_t sbyte;
            const float sdq = block_scale<FMT>(block_absmax<DT, W>(xr), ts, p.mx_rule, sbyte);
            float sq[K];
            bool dead[K];
            relaxed_scales<K>(sdq, c, d, sq, dead);
            float rho[K];
            if (want_gx) scale_ratios<K>(sdq, sq, dead, rho);
            float gd[K], gc;
            df T[K], gS;
            block_bwd<DT, B, K, false, HALF>(xr, gr, sq, dead, rho, c, d, sdq, p.ste, want_gx, true,
                                             p.gx, off, gd, gc, T, gS);
#pragma unroll
            for (int k = 0; k < K; ++k) acc[k] = df_add(acc[k], T[k]);
        }
    }
#pragma unroll
    for (int k = 0; k < K; ++k) red[threadIdx.x * K + k] = make_float2(acc[k].h, acc[k].l);
    __syncthreads();
    if (ty != 0 || !col_ok) return;
    float2* part = reinterpret_cast<float2*>(p.ws) + static_cast<size_t>(blockIdx.y) * p.nsub;
#pragma unroll
    for (int k = 0; k < K; ++k) {
        df a = acc[k];
        for (uint32_t t = 1; t < nty; ++t) {
            const float2 v = red[(t * p.tx + tx) * K + k];
            a = df_add(a, df{v.x, v.y});
        }
        part[static_cast<size_t>(cb) * K + k] = make_float2(a.h, a.l);
    }
}

// One CTA per hardware-block column j: sums the row-group partials of its K
// sub-blocks (fixed strided split, then a fixed shared-memory tree), then
// the coefficient gradients of the column.
template <int FMT, int SUB>
__global__ void __launch_bounds__(kThreads) fq_bwd_shared_finalize(const KParams p, uint32_t ny)
{
    constexpr int B = FMT == 0 ? 32 : 16;
    constexpr int K = B / SUB;
    __shared__ float sh_h[kThreads], sh_l[kThreads];
    __shared__ float res_h[K], res_l[K];
    const uint32_t j = blockIdx.x;
    const float2* part = reinterpret_cast<const float2*>(p.ws);
    for (int k = 0; k < K; ++k) {
        const uint32_t col = j * K + k;
        df a = {0.0f, 0.0f};
        for (uint32_t y = threadIdx.x; y < ny; y += kThreads) {
            const float2 v = part[static_cast<size_t>(y) * p.nsub + col];
            a = df_add(a, df{v.x, v.y});
        }
        sh_h[threadIdx.x] = a.h;
        sh_l[threadIdx.x] = a.l;
        __syncthreads();
        for (int w = kThreads / 2; w > 0; w >>= 1) {
            if (threadIdx.x < w) {
                const df s = df_add(df{sh_h[threadIdx.x], sh_l[threadIdx.x]},
                                    df{sh_h[threadIdx.x + w], sh_l[threadIdx.x + w]});
                sh_h[threadIdx.x] = s.h;
                sh_l[threadIdx.x] = s.l;
            }
            __syncthreads();
        }
        if (threadIdx.x == 0) {
            res_h[k] = sh_h[0];
            res_l[k] = sh_l[0];
        }
        __syncthreads();
    }
    if (threadIdx.x != 0) return;
    const float c = p.crs ? __ldg(p.crs + j) : 1.0f;
    float d[K];
    df T[K];
    for (int k = 0; k < K; ++k) {
        d[k] = p.dgs ? __ldg(p.dgs + j * K + k) : 1.0f;
        T[k] = df{res_h[k], res_l[k]};
    }
    float gd[K], gc;
    block_coef_grads<K>(T, c, d, gd, gc);
    if (p.gdgs)
        for (int k = 0; k < K; ++k) p.gdgs[j * K + k] = gd[k];
    if (p.gcrs) p.gcrs[j] = gc;
    if (p.step) {
        // AdamW on the shared coefficients once their gradient is complete
        const AdamW aw = adamw_setup(p);
        if (p.new_crs) {
            float m = p.opt_m[0][j], v = p.opt_v[0][j];
            p.new_crs[j] = adamw_update(c, gc, m, v, aw.step_c, aw.decay_c, aw);
            p.opt_m[0][j] = m;
            p.opt_v[0][j] = v;
        }
        if (p.new_dgs)
            for (int k = 0; k < K; ++k) {
                float m = p.opt_m[1][j * K + k], v = p.opt_v[1][j * K + k];
                p.new_dgs[j * K + k] = adamw_update(d[k], gd[k], m, v, aw.step_c, aw.decay_c, aw);
                p.opt_m[1][j * K + k] = m;
                p.opt_v[1][j * K + k] = v;
            }
    }
}

// ---------------------------------------------------------------------------
// NVFP4 per-tensor alpha (Eq. 2): per-CTA max|x| into scratch, then one CTA
// takes the max of the partials and writes fl(amax / 2688).
// ---------------------------------------------------------------------------
// max|x| over the chunks of one tensor that CTA `cta` of `n_ctas` covers
// (grid-stride), reduced over the CTA; thread 0 holds the result.
template <int DT>
__device__ __forceinline__ float alpha_cta_max(const KParams& p, uint32_t cta, uint32_t n_ctas, float* red)
{
    constexpr int U = DT != 0 ? 4 : 2;
    float m = 0.0f;
    const uint32_t span = U * kThreads;
    for (uint32_t base = cta * span; base < p.n_chunks; base += n_ctas * span) {
        ChunkRaw<DT> xr[U];
#pragma unroll
        for (int j = 0; j < U; ++j) {
            const uint32_t s = base + j * kThreads + threadIdx.x;
            if (s < p.n_chunks) {
                uint64_t off;
                if (p.strided) {
                    const uint32_t row = fast_div(s, p.div_cpr);
                    off = static_cast<uint64_t>(row) * p.ld + static_cast<uint64_t>(s - row * p.cpr) * 8u;
                } else {
                    off = static_cast<uint64_t>(s) * 8u;
                }
                load_chunk<DT>(xr[j], p.x, off);
            } else {
                zero_chunk<DT>(xr[j]);
            }
        }
#pragma unroll
        for (int j = 0; j < U; ++j) {
            float v[8];
            unpack_chunk<DT>(xr[j], v);
#pragma unroll
            for (int e = 0; e < 8; ++e) m = fmaxf(m, fabsf(v[e]));
        }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) m = fmaxf(m, __shfl_xor_sync(kFullMask, m, o));
    if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = m;
    __syncthreads();
    if (threadIdx.x < 32) {
        m = (threadIdx.x < kThreads / 32) ? red[threadIdx.x] : 0.0f;
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) m = fmaxf(m, __shfl_xor_sync(kFullMask, m, o));
    }
    return m;
}

template <int DT>
__global__ void __launch_bounds__(kThreads) alpha_partial_kernel(const KParams p)
{
    // the final reduction may be launched now: it waits for this grid to
    // complete (programmatic dependent launch) before reading the partials
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    __shared__ float red[kThreads / 32];
    const float m = alpha_cta_max<DT>(p, blockIdx.x, gridDim.x, red);
    if (threadIdx.x == 0) p.ws[blockIdx.x] = m;
}

// Group form: g.start[t] .. g.start[t + 1] are the CTAs given to tensor t
// (in proportion to its size, at least one); each writes its partial to
// g.p[0].ws[blockIdx.x].
template <int DT>
__global__ void __launch_bounds__(kThreads) alpha_group_partial_kernel(const __grid_constant__ KGroup g)
{
    __shared__ float red[kThreads / 32];
    int t = 0;
    while (t + 1 < g.n && blockIdx.x >= g.start[t + 1]) ++t;
    const float m = alpha_cta_max<DT>(g.p[t], blockIdx.x - g.start[t], g.start[t + 1] - g.start[t], red);
    if (threadIdx.x == 0) g.p[0].ws[blockIdx.x] = m;
}

}  // namespace focus
