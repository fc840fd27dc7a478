// Backward (STE) kernels, MXFP4: per-row and shared-row coefficients.
#include "fq_launch.h"

namespace focus {

cudaError_t launch_bwd_mx(int dt, int sub, const KParams& p, cudaStream_t st)
{
    const bool sfpg = p.gsfp != nullptr || p.new_sfp != nullptr;
    if (p.step) return launch_bwd_adamw_mx(dt, sub, sfpg, p, st);
    if (sfpg) return dt ? linear_by_sub<0, 1, kBwdS>(sub, p, st) : linear_by_sub<0, 0, kBwdS>(sub, p, st);
    return dt ? linear_by_sub<0, 1, kBwd>(sub, p, st) : linear_by_sub<0, 0, kBwd>(sub, p, st);
}

cudaError_t launch_bwd_shared_mx(int dt, int sub, const KParams& p, uint32_t ny, cudaStream_t st)
{
    return dt ? bwd_shared_by_sub<0, 1>(sub, p, ny, st) : bwd_shared_by_sub<0, 0>(sub, p, ny, st);
}

}  // namespace focus
