// fp4_gemm.cu -- block-scaled FP4 GEMM on the 5th-generation tensor cores
// (tcgen05), consuming focus_pack_mma exports directly:
//   D[m, n] = alpha_a * alpha_b * sum_k A[m, k] * B[n, k]       (NVFP4)
//   D[m, n] = sum_k A[m, k] * B[n, k]                           (MXFP4)
// with A[m, k] = E2M1(code) * scale(m, k / block).  This is the deployment
// the paper's "no inference overhead" refers to (Sec. 1, Sec. 3.1): only the
// exported codes and hardware scales enter the product.
//
// Persistent, warp-specialised kernel on CTA pairs (clusters of two CTAs,
// one CTA per SM), 256 x 256 tiles of D: one M = 256, N = 256 pair MMA
// (tcgen05.mma.cta_group::2) per K = 64 step, rank 0 of the pair issuing it.
// Each CTA holds 128 rows of A and 128 of the 256 rows of B in its shared
// memory and 128 rows of D in its tensor memory, so an SM loads 32 KB of
// codes per K chunk instead of the 48 KB of a one-CTA 128 x 256 tile.
//   warp 0     TMA producer (both CTAs): per K chunk of 256 elements (128
//              bytes of codes per row) the CTA's halves of the A and B tiles
//              (2D TMA, 128-byte swizzle) and the chunk's scale tiles (A: the
//              CTA's rows; B: both halves) into a ring of five stages;
//   warp 1     MMA issuer (rank 0): four K = 64 pair MMAs per chunk, then a
//              commit to the stage's empty barrier in each CTA;
//   warps 2-5  epilogue (both CTAs): accumulator -> registers (one lane
//              quarter each), alpha scaling, then 32-row x 128-byte boxes of
//              D staged in shared memory and written by TMA stores;
//   warps 6-9  scale warps (both CTAs): the chunk's scale tiles shared ->
//              tensor memory (tcgen05.st, one lane quarter each) into one of
//              four sets of scale regions, then an arrival on rank 0's
//              barrier of the chunk.
// The waits of one CTA on the other's arrivals use mbarriers at cluster
// scope; the arrivals release only shared-memory operations
// (fence.release.sync_restrict), because a full cluster-scope release also
// waits for the CTA's TMA loads in flight (0.6-1.1 us per arrival, measured)
// -- the tensor-memory stores are complete (tcgen05.wait::st) and ordered by
// tcgen05.fence before the arrival.  With four scale sets the scale warps run
// four chunks ahead of the MMAs, which hides the commit -> store -> arrival
// chain (about 0.7 us across the pair); with two they could not.
// Consecutive pairs take consecutive 256-row tiles of A with the same tile
// of B, so B is read from L2 by neighbours at about the same time.
// The producer and MMA warps run their loops converged (all lanes wait,
// lane 0 issues).  Writing the scales with tcgen05.st from their own warps
// keeps them off the tensor pipe: copied there with tcgen05.cp (12 copies per
// NVFP4 chunk) they serialise with the MMAs at about 30 ns each.  Per-lane
// row stores of D (32 rows per warp instruction) cost a third of the run
// time; the staged TMA stores write whole lines.  The 256-column accumulator
// fills half of tensor memory, the scale sets the other half, so there is
// one accumulator: the bf16 epilogue holds its whole row in registers and
// releases it before staging.
//
// Scale factors in tensor memory: one MMA step reads an A region of 4
// columns and a B region of 8, in each CTA; row m of A takes lane m % 128 of
// its CTA, column (m % 128) / 32 (so quarter q reads only column q: the scale
// warps write that one); column n of B is read by each 32-lane quarter from
// its own quarter, lane n % 32, column n / 32, in both CTAs (each CTA holds
// the scales of all 256 rows of B of the pair tile).  Lane l of every quarter
// must therefore hold, in four consecutive columns, the scale words of rows
// l, l + 32, l + 64, l + 96 of a 128-row group of B: exactly line l of a
// 128 x 4 export tile (B rows 128-255 take the next four columns).  A word
// holds consecutive K blocks in byte order: one NVFP4 step uses all four
// bytes, an MXFP4 tile feeds two steps (bytes 0-1, then bytes 2-3 through the
// scale data id).
#include <cstdint>
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <algorithm>
#include <cstring>
#include <mutex>

#include "../../include/focus_fq.h"
#include "tc_ptx.cuh"

#define FOCUS_API extern "C" __attribute__((visibility("default")))

namespace focus {
namespace {

constexpr int kTile = 128;            // rows of A (and of D) each CTA of a pair holds
constexpr int kPairM = 2 * kTile;     // M of a pair tile
constexpr int kTileN = 256;           // N of a pair tile (rows of B)
constexpr int kHalfN = kTileN / 2;    // rows of B each CTA of the pair holds
constexpr int kChunk = 128;           // K bytes (256 FP4) per stage
constexpr int kStages = 5;
constexpr int kTileBytes = kTile * kChunk;          // 16 KB of A codes
constexpr int kTileBytesB = kHalfN * kChunk;        // 16 KB of B codes (this CTA's half)
constexpr int kSfBytes = 4 * 512;                   // up to four scale tiles of A
constexpr int kSfBytesB = 2 * kSfBytes;             // the same for both 128-row halves of B
constexpr int kStageBytes = kTileBytes + kTileBytesB + kSfBytes + kSfBytesB;   // 38 KB
static_assert(kStageBytes % 1024 == 0, "swizzled tiles start on 1024-byte boundaries");
// output staging: per epilogue warp two buffers of 32 rows x 128 bytes of D
// (128-byte swizzle), written to global memory by TMA stores
constexpr int kOutBox = 32 * 128;
constexpr int kOutBufs = 2;
constexpr int kSmemBytes = kStages * kStageBytes + 4 * kOutBufs * kOutBox + 1024;   // + alignment slack
constexpr int kThreads = 320;         // producer, MMA, four epilogue warps, four scale warps
// tensor memory (the same addresses in both CTAs of a pair): the 256-column
// accumulator, then four 64-column sets of scale regions used by chunks in
// turn (set k % 4 for NVFP4, (k / 2) % 4 for MXFP4); inside a set, scale tile
// j at + 16 j (A, 4 columns) and + 16 j + 8 (B, 8 columns: B rows 0-127 of
// the pair tile in the first four, rows 128-255 in the next four -- column n
// of an N = 256 MMA is read from column n / 32).  Every region starts on an
// 8-column boundary (a scale address at an odd column faulted).
constexpr uint32_t kTmemCols = 512;
constexpr uint32_t kSfBase = kTileN;
constexpr uint32_t kSfStep = 16;
constexpr uint32_t kSfSets = 4, kSfSet = 64, kSfb = 8;
static_assert(kSfBase + kSfSets * kSfSet <= kTmemCols, "tensor memory");
static_assert(kStages > 4, "the set release waits on chunk k - 4 (see the scale warps)");
constexpr uint32_t kWaitLimit = 1u << 24;   // polls; each try_wait may suspend for a while
constexpr uint32_t kPairWarps = 8;          // arrivals per phase: four warps of each CTA

struct GemmParams {
    const uint8_t* sfa;    // scale tiles of A
    const uint8_t* sfb;    // scale tiles of B
    const float* alpha_a;  // NVFP4 per-tensor scales (device)
    const float* alpha_b;
    void* d;               // [M, ldd] fp32 or bf16
    int32_t* flag;         // set to 1 if a wait gave up
    int64_t M, N, ldd;
    uint32_t tiles_k;      // scale tiles per 128-row tile row: ceil(K / block / 4)
    uint32_t tiles_m, tiles_n;   // pair tiles: ceil(M / 256), ceil(N / 256)
    uint32_t tile_rows_b;  // 128-row scale-tile rows of B: ceil(N / 128)
    uint32_t n_steps;      // ceil(K / 64)
    int d_bf16;
    int d_vec;             // rows of D start on 16-byte boundaries: TMA stores through tma_d
};

__device__ __forceinline__ void give_up(const GemmParams& p)
{
    if (p.flag) atomicOr(p.flag, 1);
}

template <int FMT>
__global__ void __launch_bounds__(kThreads, 1)
    fp4_gemm_kernel(const __grid_constant__ CUtensorMap tma_a, const __grid_constant__ CUtensorMap tma_b,
                    const __grid_constant__ CUtensorMap tma_d, const GemmParams p)
{
    extern __shared__ uint8_t smem_raw[];
    __shared__ __align__(8) uint64_t full[kStages], empty[kStages], acc_full, acc_empty, sf_full[2 * kSfSets];
    __shared__ uint32_t tbase;
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    auto stage_a = [&](uint32_t s) { return smem + s * kStageBytes; };
    auto stage_b = [&](uint32_t s) { return smem + s * kStageBytes + kTileBytes; };
    auto stage_sfa = [&](uint32_t s) { return smem + s * kStageBytes + kTileBytes + kTileBytesB; };
    auto stage_sfb = [&](uint32_t s) { return smem + s * kStageBytes + kTileBytes + kTileBytesB + kSfBytes; };

    const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
    // rank 0 of the pair issues the pair's MMAs; both CTAs load their halves,
    // write their scale factors and drain their rows of D
    const uint32_t rank = tc::cluster_rank();
    if (threadIdx.x == 0) {
        for (int s = 0; s < kStages; ++s) {
            tc::mbar_init(&full[s], 1);
            tc::mbar_init(&empty[s], 1);   // rank 0's commit
        }
        tc::mbar_init(&acc_full, 1);
        tc::mbar_init(&acc_empty, kPairWarps);
        for (uint32_t b = 0; b < 2 * kSfSets; ++b) tc::mbar_init(&sf_full[b], kPairWarps);
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    if (warp == 0) {
        tc::tmem_alloc2(&tbase, kTmemCols);
        tc::tmem_relinquish2();
    }
    tc::tc_fence_before();
    // both CTAs' barriers initialised before either arrives on the other's
    tc::cluster_sync();
    tc::tc_fence_after();
    const uint32_t tb = tbase;
    // launched as a programmatic dependent: the set-up above overlaps the
    // previous kernel in the stream; nothing it wrote is read before this
    asm volatile("griddepcontrol.wait;" ::: "memory");
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");

    // pair tiles: u = tn * tiles_m + tm, so that consecutive pairs take
    // consecutive 256-row tiles of A with the same 256-row tile of B
    const uint32_t n_groups = p.tiles_m * p.tiles_n;
    const uint32_t group0 = blockIdx.x / 2, groups_step = gridDim.x / 2;
    const uint32_t n_chunks = (p.n_steps + 3) / 4;
    constexpr uint32_t steps_per_tile = FMT == 0 ? 2 : 1;   // K steps one scale tile covers
    // chunks per scale set: an MXFP4 chunk has two scale tiles, so a set
    // (four tiles) holds two consecutive chunks, each handed over on its own
    // barrier (sf_full[set * 2 + half]); an NVFP4 chunk fills a set alone
    constexpr uint32_t kChunksPerSet = FMT == 0 ? 2 : 1;
    constexpr uint32_t kTilesPerChunk = 4 / steps_per_tile;

    if (warp == 0) {
        // ---------------- TMA producer (both CTAs) ----------------
        // The whole warp runs the loop (converged waits); lane 0 issues.
        uint32_t s = 0, ph = 0;
        bool ok = true;
        for (uint32_t u = group0; u < n_groups && ok; u += groups_step) {
            const uint32_t tm = u % p.tiles_m, tn = u / p.tiles_m;
            const int64_t row_a = static_cast<int64_t>(tm) * kPairM + rank * kTile;
            const int64_t row_b = static_cast<int64_t>(tn) * kTileN + rank * kHalfN;
            // rows wholly past M or N are not loaded: the stale bytes only
            // reach rows or columns of D that are not stored
            const bool has_a = row_a < p.M, has_b = row_b < p.N;
            const bool hi = 2 * tn + 1 < p.tile_rows_b;   // second 128-row half of B exists
            for (uint32_t c = 0; c < n_chunks; ++c) {
                if (!__all_sync(0xffffffffu, tc::mbar_wait_cl(&empty[s], ph ^ 1, kWaitLimit))) {
                    ok = false;
                    if (lane == 0) give_up(p);
                    break;
                }
                if (lane == 0) {
                    const uint32_t steps = min(4u, p.n_steps - 4 * c);
                    const uint32_t sf_tiles = (steps + steps_per_tile - 1) / steps_per_tile;
                    const uint32_t tile0 = (4 * c) / steps_per_tile;
                    const uint32_t bytes = (has_a ? kTileBytes + sf_tiles * 512 : 0) + (has_b ? kTileBytesB : 0) +
                                           (hi ? 2 : 1) * sf_tiles * 512;
                    tc::mbar_arrive_expect_tx(&full[s], bytes);
                    if (has_b)
                        tc::tma_load_2d(stage_b(s), &tma_b, static_cast<int32_t>(c * kChunk),
                                        static_cast<int32_t>(row_b), &full[s]);
                    if (has_a) {
                        tc::tma_load_2d(stage_a(s), &tma_a, static_cast<int32_t>(c * kChunk),
                                        static_cast<int32_t>(row_a), &full[s]);
                        tc::bulk_load(stage_sfa(s),
                                      p.sfa + (static_cast<size_t>(2 * tm + rank) * p.tiles_k + tile0) * 512,
                                      sf_tiles * 512, &full[s]);
                    }
                    // the scales of both halves of B: each CTA's tensor core
                    // reads those of all 256 columns of the pair tile
                    tc::bulk_load(stage_sfb(s), p.sfb + (static_cast<size_t>(2 * tn) * p.tiles_k + tile0) * 512,
                                  sf_tiles * 512, &full[s]);
                    if (hi)
                        tc::bulk_load(stage_sfb(s) + kSfBytes,
                                      p.sfb + (static_cast<size_t>(2 * tn + 1) * p.tiles_k + tile0) * 512,
                                      sf_tiles * 512, &full[s]);
                }
                __syncwarp();
                if (++s == kStages) {
                    s = 0;
                    ph ^= 1;
                }
            }
        }
        // every stage released: no commit still to arrive on this CTA's
        // barriers when it exits
        for (int i = 0; i < kStages && ok; ++i) {
            if (!__all_sync(0xffffffffu, tc::mbar_wait_cl(&empty[s], ph ^ 1, kWaitLimit))) {
                if (lane == 0) give_up(p);
                break;
            }
            if (++s == kStages) {
                s = 0;
                ph ^= 1;
            }
        }
    } else if (warp == 1) {
        // ---------------- MMA issuer (rank 0 only) ----------------
        // The whole warp runs the loop (converged waits); lane 0 issues.
        if (rank == 0) {
            uint32_t s = 0, acc_ph = 0, k = 0;
            bool ok = true;
            for (uint32_t u = group0; u < n_groups && ok; u += groups_step) {
                // both CTAs' rows of the accumulator drained
                if (!__all_sync(0xffffffffu, tc::mbar_wait_cl(&acc_empty, acc_ph ^ 1, kWaitLimit))) {
                    if (lane == 0) give_up(p);
                    break;
                }
                tc::tc_fence_after();
                for (uint32_t c = 0; c < n_chunks; ++c) {
                    // this chunk's scales in both CTAs' tensor memory; the scale
                    // warps arrive on sf_full only after observing their stage's
                    // full barrier, so both halves of the codes are in shared
                    // memory too
                    const uint32_t pair = k / kChunksPerSet, set = pair % kSfSets;
                    const bool got = tc::mbar_wait_cl(&sf_full[set * kChunksPerSet + k % kChunksPerSet],
                                                      (pair / kSfSets) & 1u, kWaitLimit);
                    if (!__all_sync(0xffffffffu, got)) {
                        ok = false;
                        if (lane == 0) give_up(p);
                        break;
                    }
                    ++k;
                    tc::tc_fence_after();
                    if (lane == 0) {
                        const uint32_t steps = min(4u, p.n_steps - 4 * c);
                        const uint32_t sfbase =
                            tb + kSfBase + kSfSet * set + kSfStep * kTilesPerChunk * ((k - 1) % kChunksPerSet);
                        const uint32_t a0 = tc::smem_u32(stage_a(s)), b0 = tc::smem_u32(stage_b(s));
                        for (uint32_t kk = 0; kk < steps; ++kk) {
                            const uint64_t ad = tc::smem_desc_sw128(a0 + 32 * kk);
                            const uint64_t bd = tc::smem_desc_sw128(b0 + 32 * kk);
                            const uint32_t j = kk / steps_per_tile;
                            const uint32_t sfa = sfbase + kSfStep * j, sfb = sfbase + kSfb + kSfStep * j;
                            const uint32_t accumulate = (c > 0 || kk > 0) ? 1u : 0u;
                            if (FMT == 0)
                                tc::mma2_mxf4(tb, ad, bd, tc::idesc_fp4(kPairM, kTileN, true, 2 * (kk % 2)), sfa,
                                              sfb, accumulate);
                            else
                                tc::mma2_nvf4(tb, ad, bd, tc::idesc_fp4(kPairM, kTileN, false), sfa, sfb,
                                              accumulate);
                        }
                        // the stage is free in both CTAs once these MMAs are done
                        tc::mma_commit2(tc::peer_addr(&empty[s], 0));
                        tc::mma_commit2(tc::peer_addr(&empty[s], 1));
                    }
                    __syncwarp();
                    if (++s == kStages) s = 0;
                }
                if (!ok) break;
                if (lane == 0) {
                    tc::mma_commit2(tc::peer_addr(&acc_full, 0));
                    tc::mma_commit2(tc::peer_addr(&acc_full, 1));
                }
                __syncwarp();
                acc_ph ^= 1;
            }
        }
    } else if (warp >= 6) {
        // ---------------- scale warps (warps 6-9: lane quarters 2, 3, 0, 1; both CTAs) ----------------
        // Chunk k (counted over all tiles of this pair) uses stage k % kStages
        // and scale set (k / kChunksPerSet) % 4.  Before a set is rewritten,
        // the MMAs of the chunks that last used it must be complete: NVFP4
        // (one chunk per set) those of chunk k - 4; MXFP4 (pairs of chunks
        // 2 p, 2 p + 1) those of chunk 2 p - 7, implied by chunk k - 4 and
        // checked before the first chunk of the pair is written.  Rank 0's
        // commit of chunk j = k - 4 completes phase j / kStages of the empty
        // barrier of stage j % kStages in both CTAs; that barrier cannot have
        // moved on to the next phase yet (it would take the MMAs of chunk
        // j + kStages > k, which wait for these scales).
        const uint32_t q = warp % 4;
        const uint32_t lane_addr = tb + ((q * 32) << 16);
        uint32_t s = 0, ph = 0, k = 0;
        bool ok = true;
        for (uint32_t u = group0; u < n_groups && ok; u += groups_step) {
            for (uint32_t c = 0; c < n_chunks; ++c, ++k) {
                // the chunk's scale lines into registers as soon as its stage
                // has landed, before waiting for its scale set to be free
                if (!__all_sync(0xffffffffu, tc::mbar_wait_hot(&full[s], ph, kWaitLimit))) {
                    if (lane == 0) give_up(p);
                    ok = false;
                    break;
                }
                const uint32_t steps = min(4u, p.n_steps - 4 * c);
                const uint32_t sf_tiles = (steps + steps_per_tile - 1) / steps_per_tile;
                uint32_t la[kTilesPerChunk];
                uint4 lb[kTilesPerChunk], lh[kTilesPerChunk];
#pragma unroll
                for (uint32_t j = 0; j < kTilesPerChunk; ++j) {
                    if (j < sf_tiles) {
                        // A: quarter q reads only column q of the region (row q * 32 + lane)
                        la[j] = *reinterpret_cast<const uint32_t*>(stage_sfa(s) + 512 * j + 16 * lane + 4 * q);
                        lb[j] = *reinterpret_cast<const uint4*>(stage_sfb(s) + 512 * j + 16 * lane);
                        lh[j] = *reinterpret_cast<const uint4*>(stage_sfb(s) + kSfBytes + 512 * j + 16 * lane);
                    }
                }
                if (k >= 4 && (kChunksPerSet == 1 || k % 2 == 0)) {
                    const uint32_t j = k - 4;
                    if (!__all_sync(0xffffffffu,
                                    tc::mbar_wait_cl(&empty[j % kStages], (j / kStages) & 1u, kWaitLimit))) {
                        if (lane == 0) give_up(p);
                        ok = false;
                        break;
                    }
                }
                tc::tc_fence_after();
                const uint32_t set = (k / kChunksPerSet) % kSfSets;
                const uint32_t sfbase =
                    lane_addr + kSfBase + kSfSet * set + kSfStep * kTilesPerChunk * (k % kChunksPerSet);
#pragma unroll
                for (uint32_t j = 0; j < kTilesPerChunk; ++j) {
                    if (j < sf_tiles) {
                        tc::tmem_st_x1(sfbase + kSfStep * j + q, la[j]);
                        // rows 128-255 of B (stale but finite-or-not bytes when B has no
                        // such rows: they only reach columns of D that are not stored)
                        tc::tmem_st_x8(sfbase + kSfb + kSfStep * j, lb[j].x, lb[j].y, lb[j].z, lb[j].w, lh[j].x,
                                       lh[j].y, lh[j].z, lh[j].w);
                    }
                }
                tc::tmem_wait_st();
                tc::tc_fence_before();
                __syncwarp();
                if (lane == 0) tc::mbar_arrive_cl(tc::peer_addr(&sf_full[set * kChunksPerSet + k % kChunksPerSet], 0));
                if (++s == kStages) {
                    s = 0;
                    ph ^= 1;
                }
            }
        }
    } else {
        // ---------------- epilogue (warps 2-5: lane quarters 2, 3, 0, 1; both CTAs) ----------------
        const uint32_t q = warp % 4;
        const uint32_t lane_addr = tb + ((q * 32) << 16);
        const float scale = FMT == 1 ? __fmul_rn(__ldg(p.alpha_a), __ldg(p.alpha_b)) : 1.0f;
        uint32_t acc_ph = 0;
        // staging buffers of this warp; lane 0 tracks which committed bulk
        // group last read each one
        uint8_t* const obase = smem + kStages * kStageBytes + (warp - 2) * kOutBufs * kOutBox;
        uint32_t obuf = 0, ngroups = 0;
        uint32_t last_group[kOutBufs];
#pragma unroll
        for (int b = 0; b < kOutBufs; ++b) last_group[b] = 0xffffffffu;
        // the next buffer, once the store that last read it is done reading
        auto out_stage = [&](uint32_t ob) {
            const uint32_t b = ob % kOutBufs;
            if (lane == 0 && last_group[b] != 0xffffffffu) {
                if (ngroups - 1 - last_group[b] == 0) tc::bulk_wait_read<0>();
                else tc::bulk_wait_read<1>();
            }
            __syncwarp();
            return obase + b * kOutBox;
        };
        auto out_issue = [&](uint8_t* buf, int32_t x, int32_t y) {
            tc::fence_async_smem();
            __syncwarp();
            if (lane == 0 && x < p.N && y < p.M) {
                tc::tma_store_2d(&tma_d, buf, x, y);
                tc::bulk_commit();
                last_group[obuf % kOutBufs] = ngroups++;
            }
            ++obuf;
        };
        for (uint32_t u = group0; u < n_groups; u += groups_step) {
            const uint32_t tm = u % p.tiles_m, tn = u / p.tiles_m;
            const bool got = __all_sync(0xffffffffu, tc::mbar_wait_cl(&acc_full, acc_ph, kWaitLimit));
            if (!got) {
                if (lane == 0) give_up(p);
                break;
            }
            tc::tc_fence_after();
            const int64_t row0 = static_cast<int64_t>(tm) * kPairM + rank * kTile;   // this CTA's rows of D
            const int64_t m = row0 + q * 32 + lane;
            const int64_t n0 = static_cast<int64_t>(tn) * kTileN;
            if (p.d_vec) {
                // D through shared memory: per 32-row x 128-byte box, each
                // lane writes its row (16-byte chunk j of row r at chunk
                // j ^ (r % 8), the TMA 128-byte swizzle), then lane 0 issues
                // the TMA store.  Rows >= M and columns >= N are clipped by
                // the tensor map.
                const int32_t y = static_cast<int32_t>(row0) + q * 32;
                if (p.d_bf16) {
                    // the whole row of the tile in registers first, so that the
                    // accumulator is released before any staging
                    uint32_t w[kTileN / 2];
#pragma unroll
                    for (int cb = 0; cb < kTileN / 32; cb += 2) {
                        // two loads in flight per wait
                        uint32_t r[2][32];
                        tc::tmem_ld_x32(lane_addr + 32 * cb, r[0]);
                        tc::tmem_ld_x32(lane_addr + 32 * (cb + 1), r[1]);
                        tc::tmem_wait_ld();
#pragma unroll
                        for (int hb = 0; hb < 2; ++hb) {
#pragma unroll
                            for (int e = 0; e < 16; ++e) {
                                const __nv_bfloat162 h = __floats2bfloat162_rn(__fmul_rn(__uint_as_float(r[hb][2 * e]), scale),
                                                                               __fmul_rn(__uint_as_float(r[hb][2 * e + 1]), scale));
                                w[16 * (cb + hb) + e] = *reinterpret_cast<const uint32_t*>(&h);
                            }
                        }
                    }
                    tc::tc_fence_before();
                    __syncwarp();
                    if (lane == 0) tc::mbar_arrive_cl(tc::peer_addr(&acc_empty, 0));
#pragma unroll
                    for (int i = 0; i < kTileN / 64; ++i) {
                        uint8_t* buf = out_stage(obuf);
#pragma unroll
                        for (int j = 0; j < 8; ++j)
                            *reinterpret_cast<uint4*>(buf + lane * 128 + ((j ^ (lane & 7)) << 4)) =
                                make_uint4(w[32 * i + 4 * j], w[32 * i + 4 * j + 1], w[32 * i + 4 * j + 2],
                                           w[32 * i + 4 * j + 3]);
                        out_issue(buf, static_cast<int32_t>(n0) + 64 * i, y);
                    }
                } else {
#pragma unroll 1
                    for (int cb = 0; cb < kTileN / 32; ++cb) {
                        uint32_t r[32];
                        tc::tmem_ld_x32(lane_addr + 32 * cb, r);
                        tc::tmem_wait_ld();
                        if (cb == kTileN / 32 - 1) {
                            tc::tc_fence_before();
                            __syncwarp();
                            if (lane == 0) tc::mbar_arrive_cl(tc::peer_addr(&acc_empty, 0));
                        }
                        uint8_t* buf = out_stage(obuf);
#pragma unroll
                        for (int j = 0; j < 8; ++j)
                            *reinterpret_cast<float4*>(buf + lane * 128 + ((j ^ (lane & 7)) << 4)) =
                                make_float4(__fmul_rn(__uint_as_float(r[4 * j]), scale),
                                            __fmul_rn(__uint_as_float(r[4 * j + 1]), scale),
                                            __fmul_rn(__uint_as_float(r[4 * j + 2]), scale),
                                            __fmul_rn(__uint_as_float(r[4 * j + 3]), scale));
                        out_issue(buf, static_cast<int32_t>(n0) + 32 * cb, y);
                    }
                }
                acc_ph ^= 1;
                continue;
            }
#pragma unroll 1
            for (int cb = 0; cb < kTileN / 32; ++cb) {
                uint32_t r[32];
                tc::tmem_ld_x32(lane_addr + 32 * cb, r);
                tc::tmem_wait_ld();
                if (cb == kTileN / 32 - 1) {
                    // the accumulator is free once its last columns are in registers
                    tc::tc_fence_before();
                    __syncwarp();
                    if (lane == 0) tc::mbar_arrive_cl(tc::peer_addr(&acc_empty, 0));
                }
                // rows of D off 16-byte boundaries: element stores
                if (m < p.M) {
                    const int64_t nb = n0 + 32 * cb;
                    if (p.d_bf16) {
                        __nv_bfloat16* dst = static_cast<__nv_bfloat16*>(p.d) + m * p.ldd + nb;
                        for (int i = 0; i < 32 && nb + i < p.N; ++i)
                            dst[i] = __float2bfloat16_rn(__fmul_rn(__uint_as_float(r[i]), scale));
                    } else {
                        float* dst = static_cast<float*>(p.d) + m * p.ldd + nb;
                        for (int i = 0; i < 32 && nb + i < p.N; ++i) dst[i] = __fmul_rn(__uint_as_float(r[i]), scale);
                    }
                }
            }
            acc_ph ^= 1;
        }
    }
    if (warp >= 2 && warp < 6 && lane == 0) tc::bulk_wait_all();   // output stores complete
    tc::tc_fence_before();
    // no MMA, commit or arrival of the pair targets either CTA after this
    tc::cluster_sync();
    tc::tc_fence_after();
    if (warp == 0) tc::tmem_dealloc2(tb, kTmemCols);
}

// D = 0 (K = 0: every sum is empty).
__global__ void zero_kernel(void* d, int64_t M, int64_t N, int64_t ldd, int bf16)
{
    const int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
    if (i >= M * N) return;
    const int64_t m = i / N, n = i % N;
    if (bf16)
        static_cast<__nv_bfloat16*>(d)[m * ldd + n] = __float2bfloat16_rn(0.0f);
    else
        static_cast<float*>(d)[m * ldd + n] = 0.0f;
}

bool misaligned(const void* p, uintptr_t a) { return (reinterpret_cast<uintptr_t>(p) & (a - 1)) != 0; }

using EncodeTiled = CUresult (*)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                 const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                 CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiled encode_fn()
{
    static EncodeTiled fn = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        void* f = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &f, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<EncodeTiled>(f);
    });
    return fn;
}

// Tensor map of a row-major [rows, cols] matrix with row pitch `pitch`
// bytes, boxes of box_rows rows x 128 bytes, 128-byte swizzle, zero fill
// (loads) or clipping (stores) outside.
bool make_map(CUtensorMap* map, CUtensorMapDataType type, const void* base, int64_t rows, int64_t cols,
              int64_t pitch, uint32_t elem_bytes, uint32_t box_rows)
{
    EncodeTiled fn = encode_fn();
    if (!fn) return false;
    const cuuint64_t dims[2] = {static_cast<cuuint64_t>(cols), static_cast<cuuint64_t>(rows)};
    const cuuint64_t strides[1] = {static_cast<cuuint64_t>(pitch)};
    const cuuint32_t box[2] = {128u / elem_bytes, box_rows};
    const cuuint32_t estr[2] = {1, 1};
    return fn(map, type, 2, const_cast<void*>(base), dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
              CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

int device_sm_count()
{
    int dev = 0, n = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return 1;
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0) return 1;
    return n;
}

template <int FMT>
cudaError_t launch(const CUtensorMap& ma, const CUtensorMap& mb, const CUtensorMap& md, const GemmParams& p,
                   cudaStream_t st)
{
    static std::once_flag once;
    static cudaError_t attr = cudaSuccess;
    std::call_once(once, [] {
        attr = cudaFuncSetAttribute(fp4_gemm_kernel<FMT>, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemBytes);
    });
    if (attr != cudaSuccess) return attr;
    cudaLaunchConfig_t cfg = {};
    cudaLaunchAttribute at[2];
    at[0].id = cudaLaunchAttributeClusterDimension;   // CTA pairs
    at[0].val.clusterDim.x = 2;
    at[0].val.clusterDim.y = 1;
    at[0].val.clusterDim.z = 1;
    at[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    at[1].val.programmaticStreamSerializationAllowed = 1;
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = kSmemBytes;
    cfg.stream = st;
    cfg.attrs = at;
    cfg.numAttrs = 2;
    // persistent: as many pairs as are resident at once (one CTA per SM)
    static int pairs = 0;
    if (pairs <= 0) {
        int n = 0;
        cfg.gridDim = dim3(2);
        cfg.numAttrs = 1;
        if (cudaOccupancyMaxActiveClusters(&n, fp4_gemm_kernel<FMT>, &cfg) != cudaSuccess || n <= 0) {
            (void)cudaGetLastError();
            n = std::max(device_sm_count() / 2, 1);
        }
        cfg.numAttrs = 2;
        pairs = n;
    }
    const uint32_t tiles = p.tiles_m * p.tiles_n;
    cfg.gridDim = dim3(2 * std::min<uint32_t>(tiles, static_cast<uint32_t>(pairs)));
    return cudaLaunchKernelEx(&cfg, fp4_gemm_kernel<FMT>, ma, mb, md, p);
}

}  // namespace
}  // namespace focus

using namespace focus;

FOCUS_API int focus_fp4_gemm(int32_t fmt, int64_t M, int64_t N, int64_t K, const uint8_t* a_codes,
                             const uint8_t* a_scale_tiles, const float* alpha_a, const uint8_t* b_codes,
                             const uint8_t* b_scale_tiles, const float* alpha_b, void* d, int32_t d_dtype,
                             int64_t ldd, int32_t* timeout_flag, focus_stream_t stream)
{
    if (fmt != FOCUS_MXFP4 && fmt != FOCUS_NVFP4) return FOCUS_ERR_INVALID_ARG;
    if (d_dtype != FOCUS_F32 && d_dtype != FOCUS_BF16) return FOCUS_ERR_INVALID_ARG;
    if (M < 0 || N < 0 || K < 0 || ldd < N) return FOCUS_ERR_INVALID_ARG;
    // rows of codes on 16-byte boundaries (the tensor maps' pitch); a last K
    // step of 32 elements reads zero codes past K (the maps' fill) with the
    // zeroed padding of the export's scale tiles
    if (K % 32 != 0) return FOCUS_ERR_UNSUPPORTED;
    if (M > (int64_t(1) << 31) - kPairM || N > (int64_t(1) << 31) - kTileN || K > (int64_t(1) << 31))
        return FOCUS_ERR_UNSUPPORTED;
    if (M == 0 || N == 0) return FOCUS_OK;
    if (!d) return FOCUS_ERR_INVALID_ARG;
    const cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    const int bf16 = d_dtype == FOCUS_BF16;
    if (misaligned(d, bf16 ? 2 : 4) || misaligned(timeout_flag, 4)) return FOCUS_ERR_MISALIGNED;
    if (K == 0) {
        const int64_t n = M * N;
        zero_kernel<<<static_cast<unsigned>((n + 255) / 256), 256, 0, st>>>(d, M, N, ldd, bf16);
        return cudaGetLastError() == cudaSuccess ? FOCUS_OK : FOCUS_ERR_CUDA;
    }
    if (!a_codes || !b_codes || !a_scale_tiles || !b_scale_tiles) return FOCUS_ERR_INVALID_ARG;
    if (fmt == FOCUS_NVFP4 && (!alpha_a || !alpha_b)) return FOCUS_ERR_INVALID_ARG;
    if (misaligned(a_codes, 16) || misaligned(b_codes, 16) || misaligned(a_scale_tiles, 16) ||
        misaligned(b_scale_tiles, 16) || misaligned(alpha_a, 4) || misaligned(alpha_b, 4))
        return FOCUS_ERR_MISALIGNED;
    CUtensorMap ma, mb, md;
    if (!make_map(&ma, CU_TENSOR_MAP_DATA_TYPE_UINT8, a_codes, M, K / 2, K / 2, 1, kTile) ||
        !make_map(&mb, CU_TENSOR_MAP_DATA_TYPE_UINT8, b_codes, N, K / 2, K / 2, 1, kHalfN))
        return FOCUS_ERR_CUDA;
    GemmParams p;
    p.sfa = a_scale_tiles;
    p.sfb = b_scale_tiles;
    p.alpha_a = alpha_a;
    p.alpha_b = alpha_b;
    p.d = d;
    p.flag = timeout_flag;
    p.M = M;
    p.N = N;
    p.ldd = ldd;
    const int64_t block = fmt == FOCUS_MXFP4 ? 32 : 16;
    p.tiles_k = static_cast<uint32_t>((K / block + 3) / 4);
    p.tiles_m = static_cast<uint32_t>((M + kPairM - 1) / kPairM);
    p.tiles_n = static_cast<uint32_t>((N + kTileN - 1) / kTileN);
    p.tile_rows_b = static_cast<uint32_t>((N + kTile - 1) / kTile);
    p.n_steps = static_cast<uint32_t>((K + 63) / 64);
    p.d_bf16 = bf16;
    p.d_vec = !misaligned(d, 16) && (ldd * (bf16 ? 2 : 4)) % 16 == 0;
    std::memset(&md, 0, sizeof(md));
    if (p.d_vec && !make_map(&md, bf16 ? CU_TENSOR_MAP_DATA_TYPE_BFLOAT16 : CU_TENSOR_MAP_DATA_TYPE_FLOAT32, d, M, N,
                             ldd * (bf16 ? 2 : 4), bf16 ? 2 : 4, 32))
        return FOCUS_ERR_CUDA;
    const cudaError_t e = fmt == FOCUS_MXFP4 ? launch<0>(ma, mb, md, p, st) : launch<1>(ma, mb, md, p, st);
    return e == cudaSuccess ? FOCUS_OK : FOCUS_ERR_CUDA;
}
