// Backward (STE) + fused AdamW kernels, MXFP4, per-row coefficients.
#include "fq_launch.h"

namespace focus {

cudaError_t launch_bwd_adamw_mx(int dt, int sub, bool sfpg, const KParams& p, cudaStream_t st)
{
    if (sfpg) return linear_by_dt<0, kBwdSA>(dt, sub, p, st);
    return linear_by_dt<0, kBwdA>(dt, sub, p, st);
}

}  // namespace focus
