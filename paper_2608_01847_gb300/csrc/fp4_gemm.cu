// fp4_gemm.cu -- block-scaled FP4 GEMM on the 5th-generation tensor cores
// (tcgen05), consuming focus_pack_mma exports directly:
//   D[m, n] = alpha_a * alpha_b * sum_k A[m, k] * B[n, k]       (NVFP4)
//   D[m, n] = sum_k A[m, k] * B[n, k]                           (MXFP4)
// with A[m, k] = E2M1(code) * scale(m, k / block).  This is the deployment
// the paper's "no inference overhead" refers to (Sec. 1, Sec. 3.1): only the
// exported codes and hardware scales enter the product.
//
// One CTA (4 warps) per 128 x 128 tile of D; K in chunks of 256 elements
// (128 bytes of codes per row = four K = 64 MMA steps).  Per chunk the CTA
// stages the A and B code tiles in shared memory (K-major, 8 x 16-byte core
// matrices), writes the four steps' scale words to tensor memory, and one
// thread issues the MMAs; the accumulator lives in tensor memory and is read
// back once at the end.
//
// Scale factors in tensor memory (M = N = 128, one CTA): an MMA step reads a
// 4-column region; row m of A takes lane m, column m / 32; column n of B is
// read by each 32-lane quarter of the data path from its own quarter, lane
// n % 32, column n / 32.  So lane l of every quarter holds, in the region's
// four columns, the scale words of rows l, l + 32, l + 64, l + 96 -- which is
// exactly 16-byte line l of a 128 x 4 export tile.  Each word holds the
// scales of consecutive K blocks in byte order (NVFP4: four 16-element
// blocks; MXFP4: two 32-element blocks in bytes 0-1).
#include <cstdint>
#include <cuda_runtime.h>

#include "../../include/focus_fq.h"
#include "tc_ptx.cuh"

#define FOCUS_API extern "C" __attribute__((visibility("default")))

namespace focus {
namespace {

constexpr int kGemmThreads = 128;
constexpr int kTile = 128;          // M and N of one CTA
constexpr int kChunkBytes = 128;    // K bytes (256 FP4) per chunk
// tensor memory: D in columns 0-127; the scale regions of the chunk's four
// MMA steps at 128 + 16 kk (A) and 192 + 16 kk (B), each 4 columns.  An
// MMA's scale address must be aligned (a region starting at an odd column
// raises a misaligned-address error); 16-column steps keep every region on
// a 16-column boundary.
constexpr uint32_t kTmemCols = 256;
constexpr uint32_t kSfa = 128, kSfb = 192, kSfStep = 16;
constexpr uint32_t kWaitLimit = 1u << 22;

struct GemmParams {
    const uint8_t* a;      // [M, K/2] codes
    const uint8_t* sfa;    // scale tiles of A
    const uint8_t* b;      // [N, K/2] codes
    const uint8_t* sfb;    // scale tiles of B
    const float* alpha_a;  // NVFP4 per-tensor scales (device), else null
    const float* alpha_b;
    float* d;              // [M, ldd] fp32
    int32_t* flag;         // set to 1 if an MMA completion wait gave up
    int64_t M, N, K, ldd;
    uint32_t tiles_k;      // scale tiles per 128-row tile row: ceil(K / block / 4)
};

template <int FMT>
__global__ void __launch_bounds__(kGemmThreads) fp4_gemm_kernel(const GemmParams p)
{
    __shared__ __align__(1024) uint8_t sA[kTile * kChunkBytes];
    __shared__ __align__(1024) uint8_t sB[kTile * kChunkBytes];
    __shared__ __align__(8) uint64_t bar;
    __shared__ uint32_t tbase;

    const int t = threadIdx.x, warp = t / 32, lane = t % 32;
    const int64_t m0 = static_cast<int64_t>(blockIdx.y) * kTile;
    const int64_t n0 = static_cast<int64_t>(blockIdx.x) * kTile;
    const int64_t row_bytes = p.K / 2;

    if (t == 0) tc::mbar_init(&bar, 1);
    if (warp == 0) {
        tc::tmem_alloc(&tbase, kTmemCols);
        tc::tmem_relinquish();
    }
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    tc::tc_fence_before();
    __syncthreads();
    tc::tc_fence_after();
    const uint32_t tb = tbase;
    const uint32_t lane_addr = tb + (static_cast<uint32_t>(warp * 32) << 16);
    constexpr uint32_t idesc = tc::idesc_fp4(kTile, kTile, FMT == 0);

    const int64_t n_chunks = (row_bytes + kChunkBytes - 1) / kChunkBytes;
    bool ok = true;
    for (int64_t c = 0; c < n_chunks && ok; ++c) {
        const int64_t kb0 = c * kChunkBytes;
        const int64_t left = row_bytes - kb0;
        const int n_mma = static_cast<int>((left < kChunkBytes ? left : kChunkBytes) / 32);
        // ---- code tiles: thread t stages row t of A and of B ----
#pragma unroll
        for (int j = 0; j < kChunkBytes / 16; ++j) {
            uint4 va = make_uint4(0u, 0u, 0u, 0u), vb = va;
            if (j < 2 * n_mma) {
                if (m0 + t < p.M)
                    va = __ldg(reinterpret_cast<const uint4*>(p.a + (m0 + t) * row_bytes + kb0) + j);
                if (n0 + t < p.N)
                    vb = __ldg(reinterpret_cast<const uint4*>(p.b + (n0 + t) * row_bytes + kb0) + j);
            }
            const int off = (t / 8) * 1024 + j * 128 + (t % 8) * 16;
            *reinterpret_cast<uint4*>(sA + off) = va;
            *reinterpret_cast<uint4*>(sB + off) = vb;
        }
        // ---- scale words: line `lane` of the step's export tile, all quarters ----
        for (int kk = 0; kk < n_mma; ++kk) {
            const int64_t g = c * 4 + kk;                  // global K = 64 step
            const int64_t tj = FMT == 0 ? g / 2 : g;       // tile column (4 scale columns)
            const int shift = FMT == 0 ? 16 * static_cast<int>(g % 2) : 0;
            const uint4 la = __ldg(reinterpret_cast<const uint4*>(
                p.sfa + ((m0 / kTile) * p.tiles_k + tj) * 512 + 16 * lane));
            const uint4 lb = __ldg(reinterpret_cast<const uint4*>(
                p.sfb + ((n0 / kTile) * p.tiles_k + tj) * 512 + 16 * lane));
            tc::tmem_st_x4(lane_addr + kSfa + kSfStep * kk, la.x >> shift, la.y >> shift,
                           la.z >> shift, la.w >> shift);
            tc::tmem_st_x4(lane_addr + kSfb + kSfStep * kk, lb.x >> shift, lb.y >> shift,
                           lb.z >> shift, lb.w >> shift);
        }
        tc::tmem_wait_st();
        tc::fence_async_smem();
        tc::tc_fence_before();
        __syncthreads();
        tc::tc_fence_after();
        if (t == 0) {
            const uint32_t a0 = tc::smem_u32(sA), b0 = tc::smem_u32(sB);
            for (int kk = 0; kk < n_mma; ++kk) {
                const uint64_t ad = tc::smem_desc_kmajor(a0 + 256 * kk, 128, 1024);
                const uint64_t bd = tc::smem_desc_kmajor(b0 + 256 * kk, 128, 1024);
                const uint32_t acc = (c > 0 || kk > 0) ? 1u : 0u;
                const uint32_t sfa = tb + kSfa + kSfStep * kk, sfb = tb + kSfb + kSfStep * kk;
                if (FMT == 0)
                    tc::mma_mxf4(tb, ad, bd, idesc, sfa, sfb, acc);
                else
                    tc::mma_nvf4(tb, ad, bd, idesc, sfa, sfb, acc);
            }
            tc::mma_commit(&bar);
        }
        // every thread takes the same branch afterwards
        ok = __syncthreads_and(tc::mbar_wait(&bar, static_cast<uint32_t>(c & 1), kWaitLimit)) != 0;
        tc::tc_fence_after();
        if (!ok) {
            // give the MMAs in flight a second bounded chance to finish before
            // tensor memory is released
            tc::mbar_wait(&bar, static_cast<uint32_t>(c & 1), kWaitLimit);
            if (t == 0 && p.flag) atomicOr(p.flag, 1);
        }
    }

    // ---- epilogue: lane = row, column = n ----
    if (ok && n_chunks > 0) {
        const float scale = FMT == 1 ? __fmul_rn(__ldg(p.alpha_a), __ldg(p.alpha_b)) : 1.0f;
        const int64_t m = m0 + warp * 32 + lane;
#pragma unroll 1
        for (int q = 0; q < kTile / 32; ++q) {
            uint32_t r[32];
            tc::tmem_ld_x32(lane_addr + 32 * q, r);
            tc::tmem_wait_ld();
            if (m < p.M) {
                float* dst = p.d + m * p.ldd + n0 + 32 * q;
#pragma unroll
                for (int i = 0; i < 32; ++i)
                    if (n0 + 32 * q + i < p.N) dst[i] = __fmul_rn(__uint_as_float(r[i]), scale);
            }
        }
    } else if (n_chunks == 0) {
        // K = 0: D = 0
        const int64_t m = m0 + warp * 32 + lane;
        if (m < p.M)
            for (int i = 0; i < kTile; ++i)
                if (n0 + i < p.N) p.d[m * p.ldd + n0 + i] = 0.0f;
    }
    tc::tc_fence_before();
    __syncthreads();
    tc::tc_fence_after();
    if (warp == 0) tc::tmem_dealloc(tb, kTmemCols);
}

bool misaligned(const void* p, uintptr_t a) { return (reinterpret_cast<uintptr_t>(p) & (a - 1)) != 0; }

}  // namespace
}  // namespace focus

using namespace focus;

FOCUS_API int focus_fp4_gemm(int32_t fmt, int64_t M, int64_t N, int64_t K, const uint8_t* a_codes,
                             const uint8_t* a_scale_tiles, const float* alpha_a, const uint8_t* b_codes,
                             const uint8_t* b_scale_tiles, const float* alpha_b, float* d, int64_t ldd,
                             int32_t* timeout_flag, focus_stream_t stream)
{
    if (fmt != FOCUS_MXFP4 && fmt != FOCUS_NVFP4) return FOCUS_ERR_INVALID_ARG;
    if (M < 0 || N < 0 || K < 0 || ldd < N) return FOCUS_ERR_INVALID_ARG;
    if (K % 64 != 0) return FOCUS_ERR_UNSUPPORTED;
    if (M > (int64_t(1) << 31) - kTile || N > (int64_t(65535) * kTile)) return FOCUS_ERR_UNSUPPORTED;
    if (M == 0 || N == 0) return FOCUS_OK;
    if (!d || (K > 0 && (!a_codes || !b_codes || !a_scale_tiles || !b_scale_tiles)))
        return FOCUS_ERR_INVALID_ARG;
    if (fmt == FOCUS_NVFP4 && (!alpha_a || !alpha_b)) return FOCUS_ERR_INVALID_ARG;
    if (misaligned(a_codes, 16) || misaligned(b_codes, 16) || misaligned(a_scale_tiles, 16) ||
        misaligned(b_scale_tiles, 16) || misaligned(d, 4) || misaligned(alpha_a, 4) ||
        misaligned(alpha_b, 4) || misaligned(timeout_flag, 4))
        return FOCUS_ERR_MISALIGNED;
    GemmParams p;
    p.a = a_codes;
    p.sfa = a_scale_tiles;
    p.b = b_codes;
    p.sfb = b_scale_tiles;
    p.alpha_a = alpha_a;
    p.alpha_b = alpha_b;
    p.d = d;
    p.flag = timeout_flag;
    p.M = M;
    p.N = N;
    p.K = K;
    p.ldd = ldd;
    const int64_t block = fmt == FOCUS_MXFP4 ? 32 : 16;
    p.tiles_k = static_cast<uint32_t>((K / block + 3) / 4);
    const dim3 grid(static_cast<uint32_t>((N + kTile - 1) / kTile), static_cast<uint32_t>((M + kTile - 1) / kTile));
    const cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    if (fmt == FOCUS_MXFP4)
        fp4_gemm_kernel<0><<<grid, kGemmThreads, 0, st>>>(p);
    else
        fp4_gemm_kernel<1><<<grid, kGemmThreads, 0, st>>>(p);
    return cudaGetLastError() == cudaSuccess ? FOCUS_OK : FOCUS_ERR_CUDA;
}
