// fq_kernels.cuh -- CUDA kernels of the FOCUS FP4 fake-quantizer (sm_103a).
//
// Work decomposition.  A row of `cols` elements is split into chunks of 8
// consecutive elements (one 128-bit load in bf16).  One thread owns one chunk
// at a time; the B/8 lanes that hold one hardware block (4 for MXFP4's 32, 2
// for NVFP4's 16) are adjacent lanes of a warp, so the block absmax and the
// per-block coefficient-gradient sums are warp shuffles -- no shared memory,
// no atomics.  The streaming kernels walk a linear chunk index with a
// grid-stride loop sized to the resident CTAs, U chunks per thread per step
// with all loads issued before any arithmetic.
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
#pragma once

#include "fq_device.cuh"

namespace focus {

constexpr int kThreads = 256;
enum Mode { kFwd = 0, kPack = 1, kBwd = 2 };

struct KParams {
    const void* x;
    const void* g;
    void* y;
    void* gx;
    const float* crs;
    const float* dgs;
    const float* alpha;
    float* gcrs;
    float* gdgs;
    uint8_t* codes;
    uint8_t* scales;
    float* ws;            // scratch: per-CTA partials
    uint64_t ld;          // row pitch of x / y / g / gx in elements
    uint32_t n_chunks;    // rows * cols / 8
    uint32_t cpr;         // chunks per row = cols / 8
    FastDiv div_cpr;
    uint32_t rows;
    uint32_t nsub;        // sub-blocks per row = cols / sub_block
    int strided;          // ld != cols
    int shared;           // one coefficient set for all rows
    int ste;              // 0 identity, 1 clipped
    int mx_rule;          // 0 ceiling, 1 OCP floor
};

template <int FMT, int SUB>
struct Geo {
    static constexpr int B = FMT == 0 ? 32 : 16;  // hardware block (Sec. 3.1)
    static constexpr int LPB = B / 8;             // lanes per block
    static constexpr int NS = SUB < 8 ? 8 / SUB : 1;   // sub-blocks per chunk
    static constexpr int LPS = SUB > 8 ? SUB / 8 : 1;  // lanes per sub-block
    static constexpr int EPS = 8 / NS;                 // chunk elements per sub-block
    static_assert(SUB >= 2 && SUB <= B && B % SUB == 0, "sub-block must divide the block");
};

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
#pragma unroll
    for (int o = 1; o < (FMT == 0 ? 4 : 2); o <<= 1) m = fmaxf(m, __shfl_xor_sync(kFullMask, m, o));
    if (FMT == 0) {
        const int e = mx_exponent_fast(m, mx_rule);
        byte = static_cast<uint32_t>(e + 127);
        return exp2_int(e);
    }
    return nv_scale(m, ts.alpha, ts.den, ts.bd, byte);
}

__device__ __forceinline__ float chunk_absmax(const float (&v)[8])
{
    float m = 0.0f;
#pragma unroll
    for (int e = 0; e < 8; ++e) m = fmaxf(m, fabsf(v[e]));
    return m;
}

// Relaxed quantization scale per sub-block of the chunk; "dead" when S^dq or
// S^q is zero or infinite (outputs +0, no gradient).
template <int NS>
__device__ __forceinline__ void relaxed_scales(float sdq, float c, const float (&d)[NS],
                                               float (&sq)[NS], bool (&dead)[NS])
{
#pragma unroll
    for (int t = 0; t < NS; ++t) {
        sq[t] = __fmul_rn(sdq, __fmul_rn(c, d[t]));
        dead[t] = (sdq == 0.0f) || (sq[t] == 0.0f) || isinf(sq[t]);
    }
}

// Nibble mask of the live sub-blocks of a chunk (4 bits per element).
template <int NS>
__device__ __forceinline__ uint32_t live_nibbles(const bool (&dead)[NS])
{
    constexpr int EPS = 8 / NS;
    constexpr uint32_t sub_mask = EPS == 8 ? 0xffffffffu : ((1u << (4 * EPS)) - 1u);
    uint32_t m = 0u;
#pragma unroll
    for (int t = 0; t < NS; ++t) m |= dead[t] ? 0u : (sub_mask << (4 * EPS * t));
    return m;
}

// E2M1 codes (Eq. 1) of u = fl(x / S^q) for the eight elements of a chunk,
// exact: both brackets of every quotient (see make_bracket) are converted,
// and when the two code words differ on a live element the quotients are
// recomputed by IEEE division.  Dead sub-blocks get code 0.
template <int NS>
__device__ __forceinline__ uint32_t chunk_codes(const float (&v)[8], const float (&sq)[NS],
                                                const bool (&dead)[NS])
{
    constexpr int EPS = 8 / NS;
    Bracket br[NS];
    bool ok = true;
#pragma unroll
    for (int t = 0; t < NS; ++t) {
        br[t] = make_bracket(sq[t]);
        ok = ok & (dead[t] | br[t].ok);
    }
    float lo[8], hi[8];
#pragma unroll
    for (int e = 0; e < 8; ++e) {
        lo[e] = __fmul_rn(v[e], br[e / EPS].lo);
        hi[e] = __fmul_rn(v[e], br[e / EPS].hi);
    }
    const uint32_t live = live_nibbles<NS>(dead);
    uint32_t c = e2m1_pack8(lo);
    if (!ok | (((c ^ e2m1_pack8(hi)) & live) != 0u)) {
        float u[8];
#pragma unroll
        for (int e = 0; e < 8; ++e) u[e] = __fdiv_rn(v[e], sq[e / EPS]);
        c = e2m1_pack8(u);
    }
    return c & live;
}

// Clipping mask of the STE (|fl(x / S^q)| <= 6, live sub-blocks only),
// decided on the brackets and exactly when they straddle 6.
template <int NS>
__device__ __forceinline__ void chunk_clip_mask(const float (&v)[8], const float (&sq)[NS],
                                                const bool (&dead)[NS], bool (&live)[8])
{
    constexpr int EPS = 8 / NS;
    Bracket br[NS];
#pragma unroll
    for (int t = 0; t < NS; ++t) br[t] = make_bracket(sq[t]);
    bool ambiguous = false;
#pragma unroll
    for (int e = 0; e < 8; ++e) {
        const int t = e / EPS;
        const float lo = fabsf(__fmul_rn(v[e], br[t].lo));
        const float hi = fabsf(__fmul_rn(v[e], br[t].hi));
        live[e] = !dead[t] & (hi <= 6.0f);
        ambiguous = ambiguous | (!dead[t] & (!br[t].ok | ((lo <= 6.0f) != (hi <= 6.0f))));
    }
    if (ambiguous) {
#pragma unroll
        for (int e = 0; e < 8; ++e)
            live[e] = !dead[e / EPS] & (fabsf(__fdiv_rn(v[e], sq[e / EPS])) <= 6.0f);
    }
}

// STE backward of one chunk: input gradient g * rho (rho = S^dq / S^q of the
// sub-block, Sec. 3.2; rho = 0 on dead sub-blocks, and the +0 addend turns
// -0 into +0) and the per-sub-block Sum2 of mask*g*x.
template <int DT, int NS>
__device__ __forceinline__ void bwd_chunk(const float (&v)[8], const float (&gv)[8],
                                          const float (&sq)[NS], const float (&rho)[NS],
                                          const bool (&dead)[NS], int ste, bool want_gx,
                                          bool want_T, float (&gxo)[8], df (&T)[NS])
{
    constexpr int EPS = 8 / NS;
    if (ste == 1) {
        bool live[8];
        chunk_clip_mask<NS>(v, sq, dead, live);
#pragma unroll
        for (int e = 0; e < 8; ++e) {
            const int t = e / EPS;
            if (want_gx) gxo[e] = live[e] ? __fmul_rn(gv[e], rho[t]) : 0.0f;
            if (want_T) {
                const float a = live[e] ? gv[e] : 0.0f;
                const float p = __fmul_rn(a, v[e]);  // exact for bf16 inputs
                if (e % EPS == 0) T[t] = {p, 0.0f};
                else sum2_add(T[t], p);
                if (DT == 0) T[t].l = __fadd_rn(T[t].l, __fmaf_rn(a, v[e], -p));
            }
        }
        return;
    }
#pragma unroll
    for (int e = 0; e < 8; ++e) {
        const int t = e / EPS;
        if (want_gx) gxo[e] = __fmaf_rn(gv[e], rho[t], 0.0f);
        if (want_T) {
            const float p = __fmul_rn(gv[e], v[e]);  // exact for bf16 inputs
            if (e % EPS == 0) T[t] = {p, 0.0f};
            else sum2_add(T[t], p);
            if (DT == 0) T[t].l = __fadd_rn(T[t].l, __fmaf_rn(gv[e], v[e], -p));
        }
    }
    if (want_T) {
#pragma unroll
        for (int t = 0; t < NS; ++t)
            if (dead[t]) T[t] = {0.0f, 0.0f};
    }
}

// Scale ratio rho = fl(S^dq / S^q) per sub-block (0 for dead sub-blocks).
template <int NS>
__device__ __forceinline__ void scale_ratios(float sdq, const float (&sq)[NS], const bool (&dead)[NS],
                                             float (&rho)[NS])
{
#pragma unroll
    for (int t = 0; t < NS; ++t) rho[t] = dead[t] ? 0.0f : __fdiv_rn(sdq, sq[t]);
}

// ---------------------------------------------------------------------------
// Forward / pack / per-row backward over a linear chunk index.
// ---------------------------------------------------------------------------
template <int DT, int MODE>
struct Unroll {
    static constexpr int U = DT == 1 ? (MODE == kBwd ? 2 : 4) : (MODE == kBwd ? 1 : 2);
};

template <int FMT, int DT, int SUB, int MODE>
__global__ void __launch_bounds__(kThreads) fq_linear_kernel(const KParams p)
{
    using G = Geo<FMT, SUB>;
    constexpr int U = Unroll<DT, MODE>::U;
    constexpr int NS = G::NS;
    const TensorScale ts = tensor_scale<FMT>(p.alpha);
    const bool want_gx = (MODE == kBwd) && p.gx != nullptr;
    const bool want_T = (MODE == kBwd) && (p.gcrs != nullptr || p.gdgs != nullptr);
    const uint32_t span = U * kThreads;

    for (uint32_t base = blockIdx.x * span; base < p.n_chunks; base += gridDim.x * span) {
        ChunkRaw<DT> xr[U];
        ChunkRaw<DT> gr[MODE == kBwd ? U : 1];
        uint64_t off[U];
        float cv[U];
        float dv[U][NS];
        // ---- issue every load of this step first ----
#pragma unroll
        for (int j = 0; j < U; ++j) {
            const uint32_t s = base + j * kThreads + threadIdx.x;
            cv[j] = 1.0f;
#pragma unroll
            for (int t = 0; t < NS; ++t) dv[j][t] = 1.0f;
            off[j] = 0;
            if (s < p.n_chunks) {
                uint32_t cc = 0;
                if (p.strided || p.shared) {
                    const uint32_t row = fast_div(s, p.div_cpr);
                    cc = s - row * p.cpr;
                    off[j] = static_cast<uint64_t>(row) * p.ld + static_cast<uint64_t>(cc) * 8u;
                } else {
                    off[j] = static_cast<uint64_t>(s) * 8u;
                }
                load_chunk<DT>(xr[j], p.x, off[j]);
                if (MODE == kBwd) load_chunk<DT>(gr[j], p.g, off[j]);
                const uint32_t q = p.shared ? cc : s;
                if (p.crs) cv[j] = __ldg(p.crs + q / G::LPB);
                if (p.dgs) {
                    if (SUB <= 8) load_coefs<NS>(p.dgs + static_cast<size_t>(q) * NS, dv[j]);
                    else dv[j][0] = __ldg(p.dgs + q / G::LPS);
                }
            } else {
                zero_chunk<DT>(xr[j]);
                if (MODE == kBwd) zero_chunk<DT>(gr[MODE == kBwd ? j : 0]);
            }
        }
        // ---- arithmetic and stores ----
#pragma unroll
        for (int j = 0; j < U; ++j) {
            const uint32_t s = base + j * kThreads + threadIdx.x;
            const bool valid = s < p.n_chunks;
            float v[8];
            unpack_chunk<DT>(xr[j], v);
            uint32_t sbyte;
            const float sdq = block_scale<FMT>(chunk_absmax(v), ts, p.mx_rule, sbyte);
            float sq[NS];
            bool dead[NS];
            relaxed_scales<NS>(sdq, cv[j], dv[j], sq, dead);

            if (MODE != kBwd) {
                const uint32_t codes = chunk_codes<NS>(v, sq, dead);
                if (valid) {
                    if (MODE == kFwd) {
                        float q[8];
                        e2m1_unpack8(codes, q);
#pragma unroll
                        for (int e = 0; e < 8; ++e) q[e] = __fmul_rn(q[e], sdq);
                        store_chunk<DT>(p.y, off[j], q);
                    } else {
                        __stcs(reinterpret_cast<unsigned int*>(p.codes) + s, codes);
                    }
                    if (p.scales && (s % G::LPB) == 0)
                        p.scales[s / G::LPB] = static_cast<uint8_t>(sbyte);
                }
            } else {
                float gv[8];
                unpack_chunk<DT>(gr[MODE == kBwd ? j : 0], gv);
                float gxo[8];
                float rho[NS];
                df T[NS];
                if (want_gx) scale_ratios<NS>(sdq, sq, dead, rho);
                bwd_chunk<DT, NS>(v, gv, sq, rho, dead, p.ste, want_gx, want_T, gxo, T);
                if (want_gx && valid) store_chunk<DT>(p.gx, off[j], gxo);
                if (want_T) {
                    // sub-blocks wider than a chunk: combine their lanes
#pragma unroll
                    for (int o = 1; o < G::LPS; o <<= 1) T[0] = df_add(T[0], shfl_xor_df(T[0], o));
                    const float c = cv[j];
                    const float rc = rcp_approx(c);
                    df Q = {0.0f, 0.0f};
                    float gd[NS];
#pragma unroll
                    for (int t = 0; t < NS; ++t) {
                        const float d = dv[j][t];
                        const float rd = rcp_approx(d);
                        const df qk = df_div_f(T[t], d, rd);  // T_ik / c_i^k
                        gd[t] = -__fmul_rn(__fmul_rn(df_to_f(qk), rd), rc);
                        if (G::LPS == 1 || (s % G::LPS) == 0) Q = (t == 0) ? qk : df_add(Q, qk);
                    }
#pragma unroll
                    for (int o = G::LPS; o < G::LPB; o <<= 1) Q = df_add(Q, shfl_xor_df(Q, o));
                    if (valid) {
                        if (p.gdgs) {
                            if (SUB <= 8) store_coefs<NS>(p.gdgs + static_cast<size_t>(s) * NS, gd);
                            else if ((s % G::LPS) == 0) p.gdgs[s / G::LPS] = gd[0];
                        }
                        if (p.gcrs && (s % G::LPB) == 0)
                            p.gcrs[s / G::LPB] = -__fmul_rn(__fmul_rn(df_to_f(Q), rc), rc);
                    }
                }
            }
        }
    }
}

// ---------------------------------------------------------------------------
// Backward with coefficients shared by all rows.  Thread x owns column chunk
// cc = blockIdx.x * kThreads + threadIdx.x for the rows of its row group
// (rows blockIdx.y*U + k*gridDim.y*U ...), so its coefficients stay in
// registers and its T sums accumulate in registers across rows; each row
// group then writes one partial (a double-fp32 pair) per sub-block column to
// scratch, and fq_bwd_shared_finalize sums them in a fixed order.
// ---------------------------------------------------------------------------
template <int FMT, int DT, int SUB>
__global__ void __launch_bounds__(kThreads) fq_bwd_shared_kernel(const KParams p)
{
    using G = Geo<FMT, SUB>;
    constexpr int NS = G::NS;
    constexpr int U = DT == 1 ? 2 : 1;
    const TensorScale ts = tensor_scale<FMT>(p.alpha);
    const bool want_gx = p.gx != nullptr;
    const bool want_T = p.gcrs != nullptr || p.gdgs != nullptr;
    const uint32_t cc = blockIdx.x * kThreads + threadIdx.x;
    const bool col_ok = cc < p.cpr;

    float c = 1.0f;
    float d[NS];
#pragma unroll
    for (int t = 0; t < NS; ++t) d[t] = 1.0f;
    if (col_ok) {
        if (p.crs) c = __ldg(p.crs + cc / G::LPB);
        if (p.dgs) {
            if (SUB <= 8) load_coefs<NS>(p.dgs + static_cast<size_t>(cc) * NS, d);
            else d[0] = __ldg(p.dgs + cc / G::LPS);
        }
    }
    df acc[NS];
#pragma unroll
    for (int t = 0; t < NS; ++t) acc[t] = {0.0f, 0.0f};

    for (uint32_t r0 = blockIdx.y * U; r0 < p.rows; r0 += gridDim.y * U) {
        ChunkRaw<DT> xr[U], gr[U];
        uint64_t off[U];
#pragma unroll
        for (int j = 0; j < U; ++j) {
            const uint32_t r = r0 + j;
            off[j] = static_cast<uint64_t>(r) * p.ld + static_cast<uint64_t>(cc) * 8u;
            if (col_ok && r < p.rows) {
                load_chunk<DT>(xr[j], p.x, off[j]);
                load_chunk<DT>(gr[j], p.g, off[j]);
            } else {
                zero_chunk<DT>(xr[j]);
                zero_chunk<DT>(gr[j]);
            }
        }
#pragma unroll
        for (int j = 0; j < U; ++j) {
            const bool valid = col_ok && (r0 + j) < p.rows;
            float v[8], gv[8];
            unpack_chunk<DT>(xr[j], v);
            unpack_chunk<DT>(gr[j], gv);
            uint32_t sbyte;
            const float sdq = block_scale<FMT>(chunk_absmax(v), ts, p.mx_rule, sbyte);
            float sq[NS];
            bool dead[NS];
            relaxed_scales<NS>(sdq, c, d, sq, dead);
            float gxo[8];
            float rho[NS];
            df T[NS];
            if (want_gx) scale_ratios<NS>(sdq, sq, dead, rho);
            bwd_chunk<DT, NS>(v, gv, sq, rho, dead, p.ste, want_gx, want_T, gxo, T);
            if (want_gx && valid) store_chunk<DT>(p.gx, off[j], gxo);
            if (want_T) {
#pragma unroll
                for (int t = 0; t < NS; ++t) acc[t] = df_add(acc[t], T[t]);
            }
        }
    }
    if (!want_T) return;
#pragma unroll
    for (int o = 1; o < G::LPS; o <<= 1) acc[0] = df_add(acc[0], shfl_xor_df(acc[0], o));
    if (!col_ok) return;
    float2* part = reinterpret_cast<float2*>(p.ws) + static_cast<size_t>(blockIdx.y) * p.nsub;
    if (SUB <= 8) {
#pragma unroll
        for (int t = 0; t < NS; ++t) part[static_cast<size_t>(cc) * NS + t] = make_float2(acc[t].h, acc[t].l);
    } else if ((cc % G::LPS) == 0) {
        part[cc / G::LPS] = make_float2(acc[0].h, acc[0].l);
    }
}

// One CTA per hardware-block column j: sums the row-group partials of its K
// sub-blocks (fixed strided split, then a fixed shared-memory tree), then
// dL/dc^k_j = -S_k / (c_j (c^k_j)^2) and dL/dc_j = -(sum_k S_k / c^k_j) / c_j^2.
template <int FMT, int SUB>
__global__ void __launch_bounds__(kThreads) fq_bwd_shared_finalize(const KParams p, uint32_t ny)
{
    using G = Geo<FMT, SUB>;
    constexpr int K = G::B / SUB;
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
    const float rc = rcp_approx(c);
    df Q = {0.0f, 0.0f};
    for (int k = 0; k < K; ++k) {
        const float d = p.dgs ? __ldg(p.dgs + j * K + k) : 1.0f;
        const float rd = rcp_approx(d);
        const df qk = df_div_f(df{res_h[k], res_l[k]}, d, rd);
        if (p.gdgs) p.gdgs[j * K + k] = -__fmul_rn(__fmul_rn(df_to_f(qk), rd), rc);
        Q = df_add(Q, qk);
    }
    if (p.gcrs) p.gcrs[j] = -__fmul_rn(__fmul_rn(df_to_f(Q), rc), rc);
}

// ---------------------------------------------------------------------------
// NVFP4 per-tensor alpha (Eq. 2): per-CTA max|x| into scratch, then one CTA
// takes the max of the partials and writes fl(amax / 2688).
// ---------------------------------------------------------------------------
template <int DT>
__global__ void __launch_bounds__(kThreads) alpha_partial_kernel(const KParams p)
{
    constexpr int U = DT == 1 ? 4 : 2;
    __shared__ float red[kThreads / 32];
    float m = 0.0f;
    const uint32_t span = U * kThreads;
    for (uint32_t base = blockIdx.x * span; base < p.n_chunks; base += gridDim.x * span) {
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
            m = fmaxf(m, chunk_absmax(v));
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
        if (threadIdx.x == 0) p.ws[blockIdx.x] = m;
    }
}

}  // namespace focus
