// Backward (STE) kernels, NVFP4: per-row and shared-row coefficients.
#include "fq_launch.h"

namespace focus {

cudaError_t launch_bwd_nv(int dt, int sub, const KParams& p, cudaStream_t st)
{
    const bool sfpg = p.gsfp != nullptr || p.new_sfp != nullptr;
    if (p.step) return launch_bwd_adamw_nv(dt, sub, sfpg, p, st);
    if (sfpg) return dt ? linear_by_sub<1, 1, kBwdS>(sub, p, st) : linear_by_sub<1, 0, kBwdS>(sub, p, st);
    return dt ? linear_by_sub<1, 1, kBwd>(sub, p, st) : linear_by_sub<1, 0, kBwd>(sub, p, st);
}

cudaError_t launch_bwd_shared_nv(int dt, int sub, const KParams& p, uint32_t ny, cudaStream_t st)
{
    return dt ? bwd_shared_by_sub<1, 1>(sub, p, ny, st) : bwd_shared_by_sub<1, 0>(sub, p, ny, st);
}

}  // namespace focus
