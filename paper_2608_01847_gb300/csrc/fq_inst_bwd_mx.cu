// Backward (STE) kernels, MXFP4: per-row and shared-row coefficients.
#include "fq_launch.h"

namespace focus {

cudaError_t launch_bwd_mx(int dt, int sub, const KParams& p, cudaStream_t st)
{
    const bool sfpg = p.gsfp != nullptr || p.new_sfp != nullptr;
    if (p.step) return launch_bwd_adamw_mx(dt, sub, sfpg, p, st);
    if (sfpg) return linear_by_dt<0, kBwdS>(dt, sub, p, st);
    return linear_by_dt<0, kBwd>(dt, sub, p, st);
}

cudaError_t launch_bwd_shared_mx(int dt, int sub, const KParams& p, uint32_t ny, cudaStream_t st)
{
    return bwd_shared_by_dt<0>(dt, sub, p, ny, st);
}

int shared_bwd_occupancy_mx(int dt, int sub) { return shared_occ_by<0>(dt, sub); }

}  // namespace focus
