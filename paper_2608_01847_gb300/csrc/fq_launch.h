// fq_launch.h -- host-side launch helpers shared by the C-ABI layer and the
// kernel instantiation units (internal; not part of the public ABI).
#pragma once

#include <algorithm>
#include <cstdint>
#include <cuda_runtime.h>

#include "fq_kernels.cuh"

namespace focus {

// Streaming multiprocessors of the current device (cached per device id).
inline int device_sms()
{
    static int cache[64] = {0};
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) dev = 0;
    if (dev >= 0 && dev < 64 && cache[dev] > 0) return cache[dev];
    int n = 0;
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0) n = 1;
    if (dev >= 0 && dev < 64) cache[dev] = n;
    return n;
}

// CTAs of the alpha pass (and about as many for the shared-row backward's
// row groups): a fixed multiple of the SM count, so scratch sizes are a pure
// function of the descriptor and the device.
constexpr int kCtasPerSm = 8;

inline uint32_t alpha_grid(uint32_t n_chunks)
{
    const uint32_t span = 4u * kThreads;
    const uint64_t need = (static_cast<uint64_t>(n_chunks) + span - 1) / span;
    const uint64_t cap = static_cast<uint64_t>(device_sms()) * kCtasPerSm;
    return static_cast<uint32_t>(std::max<uint64_t>(1, std::min(need, cap)));
}

// Shared-row backward: block columns per CTA (a power of two from 32 to the
// CTA size, covering the row when it is short) and the number of row groups.
inline uint32_t shared_tx(uint32_t bpr)
{
    uint32_t tx = 32;
    while (tx < bpr && tx < static_cast<uint32_t>(kThreads)) tx <<= 1;
    return tx;
}

inline uint32_t shared_col_ctas(uint32_t bpr) { return (bpr + shared_tx(bpr) - 1) / shared_tx(bpr); }

// Row groups of the shared-row backward for a kernel with `occ` resident
// CTAs per SM: the grid (column CTAs x row groups) is a whole number of
// waves of resident CTAs, about kCtasPerSm per SM, so that no last wave runs
// part-empty (1216 CTAs at 3 per SM left the SMs a third idle in the last of
// 2.67 waves), and each CTA walks an equal share of the rows.
inline uint32_t shared_row_groups(uint32_t rows, uint32_t bpr, int occ)
{
    const uint32_t nty = kThreads / shared_tx(bpr);
    const uint64_t need = (static_cast<uint64_t>(rows) + nty - 1) / nty;
    const uint64_t o = static_cast<uint64_t>(std::max(occ, 1));
    const uint64_t waves = (kCtasPerSm + o - 1) / o;
    const uint64_t cap = std::max<uint64_t>(
        1, static_cast<uint64_t>(device_sms()) * o * waves / shared_col_ctas(bpr));
    return static_cast<uint32_t>(std::max<uint64_t>(1, std::min<uint64_t>({need, cap, 65535})));
}

// Resident CTAs per SM of the shared-row backward kernel (fmt, dtype, sub)
// on the current device (defined in the backward instantiation units).
int shared_bwd_occupancy(int fmt, int dt, int sub);

// Grid of a grid-stride streaming kernel: enough CTAs for the work, at most
// what is resident at once on the device -- except for large tensors (at
// least kOversubRounds rounds of resident CTAs), which get kOversub times
// that: with CTAs finishing and starting, the CTAs of an SM fall out of step
// and their load and compute phases overlap, where resident CTAs that start
// together walk the tensor in lockstep (one 2 GiB tensor, MXFP4 step: 6219
// -> 6845 GB/s; one 256 MB tensor at 27 rounds 6436 -> 6688; Llama-70B
// layer set 6781 -> 7036).  Smaller tensors keep one round: launched side
// by side on parallel branches they already overlap, and more CTAs there
// measured slower (Qwen3-4B backward at 10 rounds: 6520 -> 6331 GB/s).
constexpr uint64_t kOversub = 8;
constexpr uint64_t kOversubRounds = 16;

template <typename Kern>
inline uint32_t stream_grid(Kern kern, int& occ_cache, uint32_t n_chunks, uint32_t span)
{
    if (occ_cache <= 0) {
        int o = 0;
        if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&o, kern, kThreads, 0) != cudaSuccess || o <= 0) o = 1;
        occ_cache = o;
    }
    const uint64_t need = (static_cast<uint64_t>(n_chunks) + span - 1) / span;
    const uint64_t cap = static_cast<uint64_t>(device_sms()) * occ_cache;
    const uint64_t grid = need >= kOversubRounds * cap ? kOversub * cap : std::min(need, cap);
    return static_cast<uint32_t>(std::max<uint64_t>(1, grid));
}

// Programmatic dependent launch: the grid may be scheduled while the
// previous kernel in the stream is still running; the kernel itself waits
// (griddepcontrol.wait) for that kernel's completion before touching memory.
template <typename Kern, typename... Args>
inline cudaError_t launch_dependent(Kern kern, uint32_t grid, cudaStream_t st, const Args&... args)
{
    cudaLaunchConfig_t cfg = {};
    cudaLaunchAttribute at[1];
    at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    at[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.gridDim = dim3(grid);
    cfg.blockDim = dim3(kThreads);
    cfg.stream = st;
    cfg.attrs = at;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kern, args...);
}

template <int FMT, int DT, int SUB, int MODE, bool HALF>
cudaError_t run_block_as(const KParams& p, cudaStream_t st)
{
    static int occ = 0;
    auto kern = fq_block_kernel<FMT, DT, SUB, MODE, HALF>;
    const uint32_t grid = stream_grid(kern, occ, p.n_blocks, Span<FMT, DT, SUB, MODE>::value);
    return launch_dependent(kern, grid, st, p);
}

// The 256-bit kernel, or (rows on 16-byte boundaries) the 128-bit one.
template <int FMT, int DT, int SUB, int MODE>
cudaError_t run_block(const KParams& p, cudaStream_t st)
{
    return p.half ? run_block_as<FMT, DT, SUB, MODE, true>(p, st) : run_block_as<FMT, DT, SUB, MODE, false>(p, st);
}

// Dispatch over the sub-block size for one (format, dtype, mode).
template <int FMT, int DT, int MODE>
cudaError_t linear_by_sub(int sub, const KParams& p, cudaStream_t st)
{
    switch (sub) {
    case 2: return run_block<FMT, DT, 2, MODE>(p, st);
    case 4: return run_block<FMT, DT, 4, MODE>(p, st);
    case 8: return run_block<FMT, DT, 8, MODE>(p, st);
    case 16: return run_block<FMT, DT, 16, MODE>(p, st);
    case 32:
        if constexpr (FMT == 0) return run_block<FMT, DT, 32, MODE>(p, st);
        break;
    default: break;
    }
    return cudaErrorInvalidValue;
}

// Dispatch over the element type (0 binary32, 1 bfloat16, 2 binary16).
template <int FMT, int MODE>
cudaError_t linear_by_dt(int dt, int sub, const KParams& p, cudaStream_t st)
{
    switch (dt) {
    case 0: return linear_by_sub<FMT, 0, MODE>(sub, p, st);
    case 1: return linear_by_sub<FMT, 1, MODE>(sub, p, st);
    case 2: return linear_by_sub<FMT, 2, MODE>(sub, p, st);
    default: return cudaErrorInvalidValue;
    }
}

// Group launches: one kernel over the concatenated blocks of up to
// kMaxGroup tensors that share format, element type and sub-block size.
template <int FMT, int DT, int SUB, int MODE, bool HALF>
cudaError_t run_group_as(const KGroup& g_blocks, cudaStream_t st)
{
    static int occ = 0;
    auto kern = fq_group_kernel<FMT, DT, SUB, MODE, HALF>;
    // every tensor starts on a tile (one CTA step of blocks)
    constexpr uint32_t span = Span<FMT, DT, SUB, MODE>::value;
    KGroup g = g_blocks;
    uint32_t at = 0;
    for (int i = 0; i < g.n; ++i) {
        g.start[i] = at;
        at += (g.p[i].n_blocks + span - 1) / span;
    }
    g.start[g.n] = at;
    const uint32_t grid = stream_grid(kern, occ, at, 1);
    kern<<<grid, kThreads, 0, st>>>(g);
    return cudaGetLastError();
}

// 128-bit accesses for the whole group if any tensor's rows need them.
template <int FMT, int DT, int SUB, int MODE>
cudaError_t run_group(const KGroup& g, cudaStream_t st)
{
    bool half = false;
    for (int i = 0; i < g.n; ++i) half = half || g.p[i].half;
    return half ? run_group_as<FMT, DT, SUB, MODE, true>(g, st) : run_group_as<FMT, DT, SUB, MODE, false>(g, st);
}

template <int FMT, int DT, int MODE>
cudaError_t group_by_sub(int sub, const KGroup& g, cudaStream_t st)
{
    switch (sub) {
    case 2: return run_group<FMT, DT, 2, MODE>(g, st);
    case 4: return run_group<FMT, DT, 4, MODE>(g, st);
    case 8: return run_group<FMT, DT, 8, MODE>(g, st);
    case 16: return run_group<FMT, DT, 16, MODE>(g, st);
    case 32:
        if constexpr (FMT == 0) return run_group<FMT, DT, 32, MODE>(g, st);
        break;
    default: break;
    }
    return cudaErrorInvalidValue;
}

template <int FMT, int MODE>
cudaError_t group_by_dt(int dt, int sub, const KGroup& g, cudaStream_t st)
{
    switch (dt) {
    case 0: return group_by_sub<FMT, 0, MODE>(sub, g, st);
    case 1: return group_by_sub<FMT, 1, MODE>(sub, g, st);
    case 2: return group_by_sub<FMT, 2, MODE>(sub, g, st);
    default: return cudaErrorInvalidValue;
    }
}

// Defined in the group instantiation units.
cudaError_t launch_group_fwd(int fmt, int dt, int sub, const KGroup& g, cudaStream_t st);
cudaError_t launch_group_pack(int fmt, int dt, int sub, const KGroup& g, cudaStream_t st);
cudaError_t launch_group_bwd_mx(int dt, int sub, bool sfpg, const KGroup& g, cudaStream_t st);
cudaError_t launch_group_bwd_nv(int dt, int sub, bool sfpg, const KGroup& g, cudaStream_t st);

// Shared-row backward: the row-group kernel, then (when coefficient
// gradients or an optimizer step are wanted) the column finalisation.
template <int FMT, int SUB>
cudaError_t run_shared_finalize(const KParams& p, uint32_t ny, cudaStream_t st)
{
    fq_bwd_shared_finalize<FMT, SUB><<<p.bpr, kThreads, 0, st>>>(p, ny);
    return cudaGetLastError();
}

template <int FMT, int DT, int SUB>
cudaError_t run_bwd_shared(const KParams& p, uint32_t ny, cudaStream_t st)
{
    const dim3 grid(shared_col_ctas(p.bpr), ny);
    if (p.half) fq_bwd_shared_kernel<FMT, DT, SUB, true><<<grid, kThreads, 0, st>>>(p);
    else fq_bwd_shared_kernel<FMT, DT, SUB, false><<<grid, kThreads, 0, st>>>(p);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess || (p.gcrs == nullptr && p.gdgs == nullptr && p.step == nullptr)) return e;
    return run_shared_finalize<FMT, SUB>(p, ny, st);
}

template <int FMT, int DT>
cudaError_t bwd_shared_by_sub(int sub, const KParams& p, uint32_t ny, cudaStream_t st)
{
    switch (sub) {
    case 2: return run_bwd_shared<FMT, DT, 2>(p, ny, st);
    case 4: return run_bwd_shared<FMT, DT, 4>(p, ny, st);
    case 8: return run_bwd_shared<FMT, DT, 8>(p, ny, st);
    case 16: return run_bwd_shared<FMT, DT, 16>(p, ny, st);
    case 32:
        if constexpr (FMT == 0) return run_bwd_shared<FMT, DT, 32>(p, ny, st);
        break;
    default: break;
    }
    return cudaErrorInvalidValue;
}

template <int FMT, int DT, int SUB>
int shared_occ()
{
    static int occ = 0;
    if (occ <= 0) {
        int o = 0;
        if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&o, fq_bwd_shared_kernel<FMT, DT, SUB, false>, kThreads,
                                                          0) !=
                cudaSuccess ||
            o <= 0)
            o = 1;
        occ = o;
    }
    return occ;
}

template <int FMT, int DT>
int shared_occ_by_sub(int sub)
{
    switch (sub) {
    case 2: return shared_occ<FMT, DT, 2>();
    case 4: return shared_occ<FMT, DT, 4>();
    case 8: return shared_occ<FMT, DT, 8>();
    case 16: return shared_occ<FMT, DT, 16>();
    case 32:
        if constexpr (FMT == 0) return shared_occ<FMT, DT, 32>();
        break;
    default: break;
    }
    return 1;
}

template <int FMT>
int shared_occ_by(int dt, int sub)
{
    switch (dt) {
    case 0: return shared_occ_by_sub<FMT, 0>(sub);
    case 1: return shared_occ_by_sub<FMT, 1>(sub);
    case 2: return shared_occ_by_sub<FMT, 2>(sub);
    default: return 1;
    }
}

template <int FMT>
cudaError_t bwd_shared_by_dt(int dt, int sub, const KParams& p, uint32_t ny, cudaStream_t st)
{
    switch (dt) {
    case 0: return bwd_shared_by_sub<FMT, 0>(sub, p, ny, st);
    case 1: return bwd_shared_by_sub<FMT, 1>(sub, p, ny, st);
    case 2: return bwd_shared_by_sub<FMT, 2>(sub, p, ny, st);
    default: return cudaErrorInvalidValue;
    }
}

// Defined in the instantiation units.
cudaError_t launch_bwd_adamw_mx(int dt, int sub, bool sfpg, const KParams& p, cudaStream_t st);
cudaError_t launch_bwd_adamw_nv(int dt, int sub, bool sfpg, const KParams& p, cudaStream_t st);
cudaError_t launch_fwd(int fmt, int dt, int sub, const KParams& p, cudaStream_t st);
cudaError_t launch_pack(int fmt, int dt, int sub, const KParams& p, cudaStream_t st);
cudaError_t launch_bwd(int fmt, int dt, int sub, const KParams& p, cudaStream_t st);
cudaError_t launch_bwd_shared(int fmt, int dt, int sub, const KParams& p, uint32_t ny,
                              cudaStream_t st);
cudaError_t launch_alpha(int dt, const KParams& p, float* alpha_out, cudaStream_t st);
cudaError_t launch_alpha_group(int dt, const KGroup& g, float* alpha_out, cudaStream_t st);

}  // namespace focus
