// Backward (STE) kernels, MXFP4: per-row and shared-row coefficients.
#include "fq_launch.h"

namespace focus {

template <int FMT, int DT, int SUB>
cudaError_t run_bwd_shared(const KParams& p, uint32_t ny, cudaStream_t st)
{
    const dim3 grid(shared_col_ctas(p.bpr), ny);
    fq_bwd_shared_kernel<FMT, DT, SUB><<<grid, kThreads, 0, st>>>(p);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess || (p.gcrs == nullptr && p.gdgs == nullptr)) return e;
    fq_bwd_shared_finalize<FMT, SUB><<<p.bpr, kThreads, 0, st>>>(p, ny);
    return cudaGetLastError();
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

cudaError_t launch_bwd_mx(int dt, int sub, const KParams& p, cudaStream_t st)
{
    if (p.gsfp) return dt ? linear_by_sub<0, 1, kBwdS>(sub, p, st) : linear_by_sub<0, 0, kBwdS>(sub, p, st);
    return dt ? linear_by_sub<0, 1, kBwd>(sub, p, st) : linear_by_sub<0, 0, kBwd>(sub, p, st);
}

cudaError_t launch_bwd_shared_mx(int dt, int sub, const KParams& p, uint32_t ny, cudaStream_t st)
{
    return dt ? bwd_shared_by_sub<0, 1>(sub, p, ny, st) : bwd_shared_by_sub<0, 0>(sub, p, ny, st);
}

}  // namespace focus
